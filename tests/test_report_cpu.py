"""Sweep reporting (phase diagram and recovery frontier), host logic.

W*(L; alpha) = min { W : pass(L, W) >= alpha * p_clean } (§3 "Sweep and
reporting").  Pinned by hand-worked grids (non-monotone rows, unsorted W
axes, the alpha = 1 boundary, missing cells) and by the cells the paper
quotes for Qwen3-4B on GSM8K (tests/golden/frontier_points_qwen3_4b_gsm8k.json),
whose frontiers must agree with what the paper says about them.
"""
import json
import math
import os

import numpy as np
import pytest

from paper_2605_30574_gb300 import report as R
from paper_2605_30574_gb300.synth import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_frontier_hand_grid():
    Ls, Ws = [0, 3, 6], [0, 5, 10, 20]
    g = np.array([[0.1, 0.5, 0.8, 0.9],
                  [0.0, 0.0, 0.0, 0.2],
                  [0.9, 0.95, 0.9, 0.9]])
    # need = 0.75 * 0.9 = 0.675
    assert R.recovery_frontier(g, Ws, 0.9, 0.75) == [10, None, 0]
    # need = 0.9 * 0.2 = 0.18: row 1 first reaches it at W = 20
    assert R.recovery_frontier(g, Ws, 0.9, 0.2) == [5, 20, 0]


def test_frontier_is_the_least_qualifying_w_not_the_last_crossing():
    # the rate dips below the threshold after W = 0: W* is still 0
    assert R.recovery_frontier(np.array([[0.8, 0.2, 0.9]]), [0, 5, 10], 1.0, 0.5) == [0]


def test_frontier_with_unsorted_w_axis():
    assert R.recovery_frontier(np.array([[1.0, 0.0, 1.0]]), [10, 0, 5], 1.0, 0.5) == [5]


def test_frontier_alpha_one_boundary_and_missing_cells():
    g = np.array([[0.89, 0.9, 1.0], [math.nan, 0.95, math.nan], [math.nan] * 3])
    # alpha = 1: a rate equal to p_clean qualifies
    assert R.recovery_frontier(g, [0, 1, 2], 0.9, 1.0) == [1, 1, None]
    with pytest.raises(ValueError):
        R.recovery_frontier(g, [0, 1, 2], 0.9, 0.0)
    with pytest.raises(ValueError):
        R.recovery_frontier(g, [0, 1, 2], 0.9, 1.5)
    with pytest.raises(ValueError):
        R.recovery_frontier(g, [0, 1], 0.9, 0.5)


def test_phase_grid_and_rendering():
    rates = {(0, 0): 0.25, (0, 4): 1.0, (2, 4): 0.5}
    g = R.phase_grid(rates, [0, 2], [0, 4])
    assert g[0, 0] == 0.25 and g[0, 1] == 1.0 and math.isnan(g[1, 0]) and g[1, 1] == 0.5
    txt = R.render_grid(g, [0, 2], [0, 4], "t")
    assert txt.splitlines()[0] == "t"
    assert txt.splitlines()[2].split() == ["0", "25", "100"]
    assert txt.splitlines()[3].split() == ["2", ".", "50"]
    f = R.render_frontiers({"A": [4, None]}, [0, 2])
    assert f.splitlines()[1].split() == ["0", "4"] and f.splitlines()[2].split() == ["2", "-"]


def test_paper_quoted_points_agree_with_its_frontier_statements():
    with open(os.path.join(GOLDEN, "frontier_points_qwen3_4b_gsm8k.json")) as f:
        gd = json.load(f)

    def grid(kind):
        pts = {tuple(int(x) for x in k.split(",")): v for k, v in gd[kind].items()}
        Ls = sorted({L for L, _ in pts})
        Ws = sorted({w for _, w in pts})
        return R.phase_grid(pts, Ls, Ws), Ls, Ws

    pc = gd["p_clean"]
    N = gd["num_layers"]
    gb, Lb, Wb = grid("BLANK")
    fb = dict(zip(Lb, R.recovery_frontier(gb, Wb, pc, 0.75)))
    # BLANK's frontier at alpha = 0.75 is at W = 0 from L = N - 6 on
    assert fb[N - 6] == 0
    gz, Lz, Wz = grid("ZERO")
    fz = dict(zip(Lz, R.recovery_frontier(gz, Wz, pc, 0.75)))
    # ZERO: 48% at L = 30, W = 0 is below 0.75 * 90%; at L = 33 it matches clean
    assert fz[N - 3] == 0 and fz[30] != 0
    # reaching 87% at L = 27 (alpha = 0.87 / 0.90): ZERO needs about seven
    # times BLANK's pre-splice steps
    a = 0.87 / pc
    wb = dict(zip(Lb, R.recovery_frontier(gb, Wb, pc, a)))[27]
    wz = dict(zip(Lz, R.recovery_frontier(gz, Wz, pc, a)))[27]
    assert wb == 25 and wz == 170 and round(wz / wb) == 7


def test_decode_pass_rates_exact_and_token():
    seqs = [W.Seq(0, 0, 4, 0), W.Seq(0, 0, 1, 2), W.Seq(0, 1, 1, 2),
            W.Seq(1, 0, 4, 0), W.Seq(1, 0, 1, 2), W.Seq(1, 1, 1, 2)]
    ref = {0: 0, 1: 3}
    toks = np.array([[5, 6, 7, 8],
                     [5, 6, 7, 8],      # matches its reference
                     [5, 6, 0, 0],      # half the tokens
                     [1, 2, 3, 4],
                     [1, 2, 3, 0],      # three quarters
                     [1, 2, 3, 4]])     # matches
    ex = R.decode_pass_rates(toks, seqs, ref, "exact")
    assert ex == {(0, 1, 2): 0.5, (1, 1, 2): 0.5}
    tk = R.decode_pass_rates(toks, seqs, ref, "token")
    assert tk == {(0, 1, 2): (1.0 + 0.75) / 2, (1, 1, 2): (0.5 + 1.0) / 2}
    with pytest.raises(ValueError):
        R.decode_pass_rates(toks, seqs, ref, "bleu")


def test_sweep_cells_layout():
    seqs, ref = R.sweep_cells(3, 2, [0, 2, 4], [0, 1], num_layers=4)
    assert len(seqs) == 3 * (1 + 2 * 3 * 2)
    for p, r in ref.items():
        assert seqs[r] == W.Seq(p, 0, 4, 0)
    assert sum(1 for q in seqs if q.prompt == 1) == 13


def test_report_on_a_hand_decode():
    seqs, ref = R.sweep_cells(2, 1, [0, 2], [0, 3], num_layers=2)
    toks = np.zeros((len(seqs), 5), dtype=np.int64)
    # prompt 1's (L = 0, W = 0) cell departs from its reference
    for b, q in enumerate(seqs):
        if q.prompt == 1 and q.L == 0 and q.W == 0:
            toks[b, 3] = 9
    rep = R.report(toks, seqs, ref, [W.BLANK], [0, 2], [0, 3], [0.75, 0.5])
    c = rep["conditions"]["BLANK"]
    assert c["grid"] == [[0.5, 1.0], [1.0, 1.0]]
    assert c["frontier"]["0.75"] == [3, 0] and c["frontier"]["0.5"] == [0, 0]
