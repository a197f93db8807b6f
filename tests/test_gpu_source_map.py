"""The source map the kernels read, dumped from the device tables, against the
oracle's statement of the rule (§3 "Splice intervention"; Algorithm 1: layer
l at step t reads the donor of the cell's slot iff l >= L and t >= W, ZERO
for a ZERO slot, the clean span otherwise), byte for byte.

* the tiny sweep at every (layer, step), t = 0 .. T;
* every batch of the four model-shaped sweeps at the layer and step
  boundaries of their grids: l in {0, L - 1, L, N - 1}, t in {0, 1, W - 1,
  W, W + 1, T / 2, T}.

splice_debug_source_map on a device descriptor reads the map back from the
device tables (not from the host plan), so this checks what the kernels use.
"""
import oracle
import pytest

from paper_2605_30574_gb300 import build as B
from paper_2605_30574_gb300 import splice as S
from paper_2605_30574_gb300.sweep import model_shape
from paper_2605_30574_gb300.synth import workloads as WL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


def _expected(wl, seqs, l, t):
    return bytes(oracle.splice_source(q.L, q.W, q.slot, wl.slot_kinds[q.slot], l, t) for q in seqs)


def _device_desc(wl, seqs, p0):
    return S.splice_desc_create(model_shape(wl), wl.num_prompts, wl.prompt_len, wl.slot_kinds,
                                [(q.prompt - p0, q.slot, q.L, q.W) for q in seqs], wl.max_steps)


def test_tiny_every_layer_and_step():
    wl = WL.get("tiny")
    seqs = wl.sequences()
    d = _device_desc(wl, seqs, 0)
    assert d.on_device
    for t in range(wl.max_steps + 1):
        for l in range(wl.num_layers):
            got = S.splice_debug_source_map(d, l, t)
            assert got == _expected(wl, seqs, l, t), (l, t)
    d.close()


@pytest.mark.parametrize("name", ["qwen3-4b", "llama3-8b", "gemma3-4b", "qwen3-8b-ladder"])
def test_model_sweeps_at_grid_boundaries(name):
    wl = WL.get(name)
    N, T = wl.num_layers, wl.max_steps
    layers = sorted({x for L in wl.L_values for x in (L - 1, L) if 0 <= x < N} | {0, N - 1})
    steps = sorted({x for W in wl.W_values for x in (W - 1, W, W + 1) if 0 <= x <= T} | {0, 1, T // 2, T})
    all_seqs = wl.sequences()
    checked = 0
    for b in range(wl.num_batches()):
        lo, hi = wl.batch_range(b)
        seqs = all_seqs[lo:hi]
        p0 = min(q.prompt for q in seqs)
        d = _device_desc(wl, seqs, p0)
        for l in layers:
            for t in steps:
                got = S.splice_debug_source_map(d, l, t)
                assert got == _expected(wl, seqs, l, t), (name, b, l, t)
                checked += 1
        d.close()
    assert checked == wl.num_batches() * len(layers) * len(steps)
