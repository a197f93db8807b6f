"""The fp64 oracle over many (sequence, layer, step) units in a process pool
(test infrastructure).  Workers are started with ``spawn`` (never forked from
a process that holds a CUDA context) and import numpy only; units are handed
out grouped by (prompt, layer) so each worker regenerates few prompt spans.
"""
from __future__ import annotations

import multiprocessing as mp
import os


def _run(args):
    name, units = args
    import oracle
    from paper_2605_30574_gb300.synth import workloads as WL
    from parity_util import CachedInputs
    wl = WL.get(name)
    inp = CachedInputs(wl)
    seqs = wl.sequences()
    return [(u, oracle.decode_attn(wl, inp, u[0], seqs[u[0]], u[1], u[2])) for u in units]


def oracle_outputs(name: str, units, workers: int = 0) -> dict:
    """{(s, l, t): oracle output [Hq][d]} for every unit (global sequence s)."""
    from paper_2605_30574_gb300.synth import workloads as WL
    wl = WL.get(name)
    seqs = wl.sequences()
    units = sorted(set(units), key=lambda u: (seqs[u[0]].prompt, u[1], u[0], u[2]))
    n = workers or max(1, min(16, len(os.sched_getaffinity(0))))
    n = min(n, len(units)) or 1
    per = -(-len(units) // n)
    chunks = [(name, units[i:i + per]) for i in range(0, len(units), per)]
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ.setdefault(k, "1")
    ctx = mp.get_context("spawn")
    with ctx.Pool(len(chunks)) as pool:
        out = {}
        for part in pool.map(_run, chunks):
            out.update(dict(part))
    return out
