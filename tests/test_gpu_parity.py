"""Parity of the CUDA path (through the C ABI) with the CPU fp64 oracle.

* the tiny sweep, exhaustively: every sequence, layer and step 0..T;
* the hand-derived cases of tests/golden/hand_cases.json, zero-padded to d = 64;
* edge shapes: ragged prompt spans, group sizes 1/2/3/4/6/8, d = 64/128/256,
  sliding windows shorter than the prompt span, a single sequence;
* the four model-shaped sweeps at full size, in the launch configuration the
  bench times, on sampled (sequence, layer, step) outputs.
"""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2605_30574_gb300 import build as B
from paper_2605_30574_gb300 import splice as S
from paper_2605_30574_gb300.sweep import SweepBatch
from paper_2605_30574_gb300.synth import host as H
from paper_2605_30574_gb300.synth import workloads as WL
from parity_util import CachedInputs, assert_close

pytestmark = pytest.mark.gpu
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


class SeqInputs:
    """Oracle inputs of a SweepBatch built from an explicit sequence list:
    sequence index s of the batch is generator sequence s."""

    def __init__(self, wl):
        self.c = CachedInputs(wl)

    def __getattr__(self, k):
        return getattr(self.c, k)


def oracle_rows(wl, inputs, seqs, l, t, which):
    return np.stack([oracle.decode_attn(wl, inputs, s, seqs[s], l, t) for s in which])


def test_tiny_exhaustive():
    wl = WL.get("tiny")
    sb = SweepBatch(wl, 0)
    inp = CachedInputs(wl)
    worst = (0.0, 0.0)
    for t in range(0, wl.max_steps + 1):
        for l in range(wl.num_layers):
            out = sb.run(l, t).cpu().numpy()
            ref = oracle_rows(wl, inp, sb.seqs, l, t, range(sb.B))
            a, r = assert_close(out, ref, f"tiny l={l} t={t}")
            worst = (max(worst[0], a), max(worst[1], r))
    S.splice_check_device_error(sb.desc)
    print("tiny exhaustive worst abs/rel", worst)


def test_tiny_zero_span_empty_suffix_is_exactly_zero():
    wl = WL.get("tiny")
    sb = SweepBatch(wl, 0)
    for l in range(wl.num_layers):
        out = sb.run(l, 0).cpu().numpy()
        m = S.splice_debug_source_map(sb.desc, l, 0)
        zero = [s for s in range(sb.B) if m[s] == S.SRC_ZERO]
        assert zero, "the tiny sweep has ZERO cells spliced at step 0"
        assert np.all(out[zero] == 0.0)


# --------------------------------------------------------------------------
# hand-derived cases on the GPU (head_dim padded with zeros to 64)
# --------------------------------------------------------------------------
KIND = {"ZERO": WL.ZERO, "BLANK": WL.BLANK, "SAME_ALGO": WL.SAME_ALGO, "DIFF_ALGO": WL.DIFF_ALGO,
        "DIFF_FAMILY": WL.DIFF_FAMILY}


def _pad(a, d=64):
    a = np.asarray(a, dtype=np.float32)
    out = np.zeros(a.shape[:-1] + (d,), np.float32)
    out[..., : a.shape[-1]] = a
    return torch.from_numpy(out).to(torch.bfloat16).cuda()


def _hand_cases():
    with open(os.path.join(GOLDEN, "hand_cases.json")) as fh:
        return json.load(fh)["cases"]


@pytest.mark.parametrize("case", _hand_cases(), ids=lambda c: c["name"])
def test_hand_cases_on_gpu(case):
    from fractions import Fraction
    kinds = tuple(KIND[k] for k in case["slot_kinds"])
    wl = WL.Workload("hand", case["num_layers"], case["num_q_heads"], case["num_kv_heads"], 64, 1,
                     case["prompt_len"], kinds, case["max_steps"], (0,), (0,), 0, 0, batch=1,
                     sliding_window=case["sliding_window"], global_every=case["global_every"],
                     sm_scale=math.log(2.0))
    seqs = [WL.Seq(0, qd["slot"], qd["L"], qd["W"]) for qd in case["queries"]]
    sb = SweepBatch(wl, seqs=seqs, fill=False)
    for l in range(wl.num_layers):
        sb.k_clean[0, l] = _pad(case["clean_k"])
        sb.v_clean[0, l] = _pad(case["clean_v"])
        st = 0
        for k, kind in enumerate(kinds):
            if kind != WL.ZERO:
                sb.k_donor[0, st, l] = _pad(case["donor_k"][str(k)])
                sb.v_donor[0, st, l] = _pad(case["donor_v"][str(k)])
                st += 1
        sb.k_suffix[:, l] = _pad(case["suffix_k"])[None]
        sb.v_suffix[:, l] = _pad(case["suffix_v"])[None]
    sb.q.copy_(_pad(case["q"])[None].expand_as(sb.q))
    d0 = len(case["q"][0])
    for i, qd in enumerate(case["queries"]):
        sb.attn(qd["l"], qd["t"])
        got = sb.out[i].cpu().numpy()
        want = np.array([[float(Fraction(x)) for x in row] for row in qd["expected"]])
        np.testing.assert_allclose(got[:, :d0], want, rtol=5e-3, atol=5e-3, err_msg=qd["why"])
        assert np.all(got[:, d0:] == 0.0)


# --------------------------------------------------------------------------
# edge shapes
# --------------------------------------------------------------------------
EDGE = [
    # name, N, Hq, Hkv, d, P, Tp, kinds, T, window, global_every
    ("ragged_tp_g4_d128", 3, 8, 2, 128, 2, 300, (WL.BLANK, WL.ZERO, WL.SAME_ALGO), 9, 0, 0),
    ("g1_d64_tp_1", 2, 4, 4, 64, 1, 1, (WL.ZERO, WL.DIFF_FAMILY), 5, 0, 0),
    ("g2_d256_window", 4, 4, 2, 256, 2, 200, (WL.BLANK, WL.ZERO), 40, 150, 3),
    ("g8_d128", 2, 16, 2, 128, 1, 129, (WL.DIFF_ALGO, WL.ZERO), 6, 0, 0),
    ("g3_d64_long", 2, 6, 2, 64, 1, 1100, (WL.BLANK,), 700, 0, 0),
    ("window_below_suffix", 3, 8, 2, 64, 1, 64, (WL.ZERO, WL.BLANK), 50, 20, 0),
    # five prompt-span splits: four of 3072 keys and a short last one
    ("long_span_5_splits", 1, 4, 2, 64, 1, 13000, (WL.SAME_ALGO, WL.ZERO), 3, 0, 0),
    # generated-span pass at every (d, rows per item) it is built for, with
    # generated spans long enough for several key splits and a ragged block:
    # one row per item at d = 128 and 256 (fewer logits per key group than
    # lanes), two rows (G = 6: three row chunks), four rows at d = 256
    ("g1_d128_long_suffix", 2, 4, 4, 128, 1, 150, (WL.BLANK, WL.ZERO), 150, 0, 0),
    ("g6_d128_long_suffix", 2, 12, 2, 128, 1, 97, (WL.DIFF_ALGO, WL.ZERO), 150, 0, 0),
    ("g4_d256_long_suffix", 2, 8, 2, 256, 1, 140, (WL.SAME_ALGO, WL.ZERO), 150, 0, 0),
    ("g1_d256_long_suffix", 2, 2, 2, 256, 1, 90, (WL.DIFF_FAMILY, WL.ZERO), 150, 0, 0),
]


@pytest.mark.parametrize("spec", EDGE, ids=lambda e: e[0])
def test_edge_shapes(spec):
    name, N, Hq, Hkv, d, P, Tp, kinds, T, win, gev = spec
    Ls = tuple(sorted({0, 1, N // 2, N}))
    Ws = tuple(sorted({0, 1, T // 2, T + 1}))
    wl = WL.Workload(name, N, Hq, Hkv, d, P, Tp, kinds, T, Ls, Ws, min(4, Tp), min(2, Tp), batch=10 ** 6,
                     sliding_window=win, global_every=gev)
    sb = SweepBatch(wl, 0)
    inp = CachedInputs(wl)
    steps = sorted({0, 1, 2, T // 2, T // 2 + 1, T})
    for t in steps:
        for l in range(N):
            out = sb.run(l, t).cpu().numpy()
            ref = oracle_rows(wl, inp, sb.seqs, l, t, range(sb.B))
            assert_close(out, ref, f"{name} l={l} t={t}")
    S.splice_check_device_error(sb.desc)


def test_single_sequence_batch():
    wl = WL.get("tiny")
    seqs = [WL.Seq(1, 0, 2, 4)]
    sb = SweepBatch(wl, seqs=seqs)
    inp = SeqInputs(wl)
    for t in (1, 3, 4, 16):
        for l in range(wl.num_layers):
            out = sb.run(l, t).cpu().numpy()
            ref = oracle_rows(wl, inp, seqs, l, t, [0])
            assert_close(out, ref, f"l={l} t={t}")


# --------------------------------------------------------------------------
# full-size sweeps, sampled
# --------------------------------------------------------------------------
def sample_points(wl, seqs, max_points=48, seed=0):
    """(s, l, t) triples around every cutoff and onset, every donor kind."""
    rng = np.random.default_rng(seed)
    N, T = wl.num_layers, wl.max_steps
    prompts = sorted({q.prompt for q in seqs})
    pick_prompts = {prompts[0], prompts[-1]}
    pts = []
    for s, q in enumerate(seqs):
        if q.prompt not in pick_prompts:
            continue
        layers = {x for x in (q.L - 1, q.L, N - 1) if 0 <= x < N}
        steps = {x for x in (1, q.W - 1, q.W, q.W + 1, T // 2, T) if 1 <= x <= T}
        for l in layers:
            for t in steps:
                pts.append((s, l, t))
    rng.shuffle(pts)
    # keep every donor slot represented
    chosen, seen = [], set()
    for p in pts:
        k = seqs[p[0]].slot
        if k not in seen:
            chosen.append(p)
            seen.add(k)
    for p in pts:
        if len(chosen) >= max_points:
            break
        if p not in chosen:
            chosen.append(p)
    return chosen


@pytest.mark.parametrize("name", ["qwen3-4b", "llama3-8b", "gemma3-4b", "qwen3-8b-ladder"])
def test_full_size_sampled(name):
    wl = WL.get(name)
    torch.cuda.empty_cache()
    sb = SweepBatch(wl, 0)
    inp = CachedInputs(wl)
    pts = sample_points(wl, sb.seqs)
    by_lt = {}
    for s, l, t in pts:
        by_lt.setdefault((l, t), []).append(s)
    got = {}
    for (l, t), ss in sorted(by_lt.items(), key=lambda kv: (kv[0][1], kv[0][0])):
        out = sb.run(l, t)
        rows = out[torch.tensor(ss, device="cuda")].cpu().numpy()
        for s, r in zip(ss, rows):
            got[(s, l, t)] = r
    S.splice_check_device_error(sb.desc)
    sb.close()
    del sb
    torch.cuda.empty_cache()
    worst = (0.0, 0.0)
    for (s, l, t), g in sorted(got.items(), key=lambda kv: (kv[0][1], kv[0][0])):
        ref = oracle.decode_attn(wl, inp, s, wl.sequences()[s], l, t)
        a, r = assert_close(g, ref, f"{name} s={s} l={l} t={t}")
        worst = (max(worst[0], a), max(worst[1], r))
    print(name, "points", len(got), "worst abs/rel", worst)


@pytest.mark.parametrize("name", ["qwen3-8b-ladder"])
def test_ladder_first_and_last_prompt_every_cell(name):
    """The sampling plan for the donor-noise ladder: every cell of the first
    and the last prompt -- prompt 0 in batch 0, prompt P - 1 in the last,
    ragged batch of 128 sequences -- at steps {1, W - 1, W, W + 1, T / 2, T}
    and layers {0, L - 1, L, N - 1} around the cell's own onset and cutoff,
    in the launch configuration the bench times (whole batches)."""
    from oracle_pool import oracle_outputs
    wl = WL.get(name)
    N, T = wl.num_layers, wl.max_steps
    seqs = wl.sequences()
    units = []
    for s, q in enumerate(seqs):
        if q.prompt not in (0, wl.num_prompts - 1):
            continue
        layers = {x for x in (0, q.L - 1, q.L, N - 1) if 0 <= x < N}
        steps = {x for x in (1, q.W - 1, q.W, q.W + 1, T // 2, T) if 1 <= x <= T}
        units += [(s, l, t) for l in layers for t in steps]
    batches = sorted({s // wl.batch for s, _, _ in units})
    assert batches == [0, wl.num_batches() - 1]
    assert wl.batch_range(batches[-1])[1] - wl.batch_range(batches[-1])[0] == 128
    got = {}
    for b in batches:
        torch.cuda.empty_cache()
        sb = SweepBatch(wl, b)
        lo = sb.s0
        by_lt = {}
        for s, l, t in units:
            if lo <= s < lo + sb.B:
                by_lt.setdefault((l, t), []).append(s)
        for (l, t), ss in sorted(by_lt.items(), key=lambda kv: (kv[0][1], kv[0][0])):
            out = sb.run(l, t)
            rows = out[torch.tensor([s - lo for s in ss], device="cuda")].cpu().numpy()
            for s, r in zip(ss, rows):
                got[(s, l, t)] = r
        S.splice_check_device_error(sb.desc)
        sb.close()
        del sb
    torch.cuda.empty_cache()
    ref = oracle_outputs(name, units)
    worst = (0.0, 0.0)
    for u in sorted(got):
        a, r = assert_close(got[u], ref[u], f"{name} s={u[0]} l={u[1]} t={u[2]}")
        worst = (max(worst[0], a), max(worst[1], r))
    print(name, "units", len(got), "worst abs/rel", worst)


# --------------------------------------------------------------------------
# softmax scale: sign and zero
# --------------------------------------------------------------------------
@pytest.mark.parametrize("scale", [-0.7, 0.0, 2.5])
def test_softmax_scale_sign_and_zero(scale):
    """sm_scale < 0 makes the largest scaled logit the smallest raw one (the
    kernels then track block minima); 0 gives uniform weights over the visible
    keys; a large positive scale sharpens the weights so the lazily moved
    reference max moves more often."""
    wl = WL.Workload(f"scale{scale}", 3, 8, 2, 128, 2, 300, (WL.BLANK, WL.ZERO, WL.SAME_ALGO), 9,
                     (0, 1, 3), (0, 2, 10), 4, 2, batch=10 ** 6, sm_scale=scale)
    sb = SweepBatch(wl, 0)
    inp = CachedInputs(wl)
    for t in (1, 2, 9):
        for l in range(wl.num_layers):
            out = sb.run(l, t).cpu().numpy()
            ref = oracle_rows(wl, inp, sb.seqs, l, t, range(sb.B))
            assert_close(out, ref, f"scale {scale} l={l} t={t}")
    S.splice_check_device_error(sb.desc)
