"""Shared helpers of the GPU parity tests: the tolerance of the path (bf16
inputs, fp32 accumulation: max abs error <= 1e-2 per element and max relative
error <= 2e-2 per output row, relative to the row's largest oracle value) and
a caching view of the host input generator for the oracle."""
from functools import lru_cache

import numpy as np

from paper_2605_30574_gb300.synth import host as H

TOL_ABS = 1e-2
TOL_REL = 2e-2


def row_errors(gpu, ref):
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    diff = np.abs(gpu - ref)
    rel = diff.max(axis=-1) / np.maximum(np.abs(ref).max(axis=-1), 1e-6)
    return float(diff.max()), float(rel.max())


def assert_close(gpu, ref, what=""):
    a, r = row_errors(gpu, ref)
    assert a <= TOL_ABS and r <= TOL_REL, f"{what}: max abs {a:.3e}, max rel {r:.3e}"
    return a, r


class CachedInputs:
    """SynthInputs with the prompt spans cached per (prompt, layer[, slot])."""

    def __init__(self, wl):
        self.g = H.SynthInputs(wl)
        self.clean_kv = lru_cache(maxsize=64)(self.g.clean_kv)
        self.donor_kv = lru_cache(maxsize=64)(self.g.donor_kv)

    def q(self, s, t, l):
        return self.g.q(s, t, l)

    def suffix_kv(self, s, l, i0, i1):
        return self.g.suffix_kv(s, l, i0, i1)
