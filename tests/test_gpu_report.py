"""Sweep reporting on a real decode sweep: a random-initialised decoder's
greedy splice-intervention decode of every (donor, L, W) cell, every decode
attention through the library, scored against each prompt's unintervened
decode (§3 "Sweep and reporting").

What must hold whatever the weights: a cell that patches no layer (L = N) or
never reaches its onset (W >= the steps generated) is the unintervened decode
token for token, so its rate is 1 and its frontier is the least W; and a cell
with onset W emits the unintervened tokens y_0 .. y_{W-1}, since no layer is
patched before step W.
"""
import numpy as np
import pytest

from paper_2605_30574_gb300 import build as B
from paper_2605_30574_gb300 import report as R
from paper_2605_30574_gb300.model import tiny_dims
from paper_2605_30574_gb300.synth import workloads as WL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


def test_decode_sweep_report_invariants():
    dims = tiny_dims()
    N = dims.num_layers
    kinds = [WL.BLANK, WL.ZERO, WL.SAME_ALGO, WL.DIFF_FAMILY]
    Ls, Ws, steps = list(range(N + 1)), [0, 1, 3, 6, 10], 10
    toks, seqs, ref = R.run_decode_sweep(dims, kinds, Ls, Ws, num_prompts=3, prompt_len=40, steps=steps, seed=2,
                                         scaffold_head=4, scaffold_tail=2, filler=3)
    assert toks.shape == (len(seqs), steps)
    for b, q in enumerate(seqs):
        r = toks[ref[q.prompt]]
        # nothing is patched before step W: y_0 .. y_{W-1} are the reference's
        w = min(max(q.W, 1), steps)
        assert np.array_equal(toks[b, :w], r[:w]), q
        if q.L >= N or q.W >= steps:
            assert np.array_equal(toks[b], r), q
    rep = R.report(toks, seqs, ref, kinds, Ls, Ws, [0.5, 1.0])
    for name, c in rep["conditions"].items():
        g = np.array([[np.nan if x is None else x for x in row] for row in c["grid"]])
        assert g.shape == (len(Ls), len(Ws)) and not np.isnan(g).any()
        assert (g[Ls.index(N)] == 1.0).all() and (g[:, Ws.index(10)] == 1.0).all(), name
        for a in ("0.5", "1.0"):
            f = c["frontier"][a]
            assert f[Ls.index(N)] == 0
            # every row reaches the threshold by the never-reached onset
            assert all(x is not None and x <= 10 for x in f)
            # W* is the least qualifying W of its row
            for i, x in enumerate(f):
                assert g[i, Ws.index(x)] >= float(a) and all(g[i, j] < float(a) for j, wv in enumerate(Ws) if wv < x)
    for name, c in rep["conditions"].items():
        g = np.array(c["grid"], dtype=np.float64)
        print(R.render_grid(g, Ls, Ws, name))
