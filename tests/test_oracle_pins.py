"""Pins of the CPU fp64 oracle against what the paper and the mathematics fix.

* the hand-enumerated splice rule table (§3, Algorithm 1) and a literal,
  in-place simulation of Algorithm 1's cache mutation;
* hand-derived outputs of tiny cases (tests/golden/hand_cases.json);
* the ZERO closed form (Table 1: all-zero K and V give logit 0 and value 0);
* torch's CPU scaled_dot_product_attention (fp64) over explicitly built caches;
* the log-sum-exp merge against single-pass softmax;
* W = 0 and W = 1 runs, donor == clean runs, monotonicity of the rule;
* planted mistakes in the oracle that these pins must catch.
"""
import json
import math
import os
from dataclasses import dataclass
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle
from oracle import splice_oracle as so
from paper_2605_30574_gb300.synth import host as H
from paper_2605_30574_gb300.synth import workloads as WL

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
KIND = {"ZERO": WL.ZERO, "BLANK": WL.BLANK, "SAME_ALGO": WL.SAME_ALGO,
        "DIFF_ALGO": WL.DIFF_ALGO, "DIFF_FAMILY": WL.DIFF_FAMILY}


# --------------------------------------------------------------------------
# helpers
# --------------------------------------------------------------------------
@dataclass
class Shape:
    num_layers: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    prompt_len: int
    max_steps: int
    slot_kinds: tuple
    sliding_window: int = 0
    global_every: int = 0
    sm_scale: float = 1.0


@dataclass
class Cell:
    prompt: int
    slot: int
    L: int
    W: int


def to_bf16(a):
    return H.f32_to_bf16_rne(np.asarray(a, dtype=np.float32))


class ArrayInputs:
    """Inputs given as explicit arrays, the same at every layer, step and prompt."""

    def __init__(self, q, ck, cv, dk, dv, sk, sv):
        self._q, self._ck, self._cv = to_bf16(q), to_bf16(ck), to_bf16(cv)
        self._dk = {int(k): to_bf16(v) for k, v in dk.items()}
        self._dv = {int(k): to_bf16(v) for k, v in dv.items()}
        self._sk, self._sv = to_bf16(sk), to_bf16(sv)

    def q(self, s, t, l):
        return self._q

    def clean_kv(self, p, l):
        return self._ck, self._cv

    def donor_kv(self, p, k, l):
        return self._dk[k], self._dv[k]

    def suffix_kv(self, s, l, i0, i1):
        return self._sk[:, i0:i1], self._sv[:, i0:i1]


class RandomInputs:
    """Random bf16 inputs per (layer, step), for cross-checks on tiny shapes."""

    def __init__(self, shp: Shape, n_donor_slots: int, seed: int):
        rng = np.random.default_rng(seed)
        N, Hq, Hkv, d, Tp, T = (shp.num_layers, shp.num_q_heads, shp.num_kv_heads,
                                shp.head_dim, shp.prompt_len, shp.max_steps)
        self.Q = to_bf16(rng.normal(0, 1, (T + 1, N, Hq, d)))
        self.CK = to_bf16(rng.normal(0, 1, (N, Hkv, Tp, d)) * 2)
        self.CV = to_bf16(rng.normal(0, 1, (N, Hkv, Tp, d)))
        self.DK = to_bf16(rng.normal(0, 1, (n_donor_slots, N, Hkv, Tp, d)) * 2)
        self.DV = to_bf16(rng.normal(0, 1, (n_donor_slots, N, Hkv, Tp, d)))
        self.SK = to_bf16(rng.normal(0, 1, (N, Hkv, T, d)))
        self.SV = to_bf16(rng.normal(0, 1, (N, Hkv, T, d)))

    def q(self, s, t, l):
        return self.Q[t, l]

    def clean_kv(self, p, l):
        return self.CK[l], self.CV[l]

    def donor_kv(self, p, k, l):
        return self.DK[k, l], self.DV[k, l]

    def suffix_kv(self, s, l, i0, i1):
        return self.SK[l, :, i0:i1], self.SV[l, :, i0:i1]


def alg1_span_by_layer(N, T, L, W):
    """Literal simulation of Algorithm 1's cache mutation.

    Returns state[(l, t)] in {'C', 'D'}: which prompt span the cache holds
    at layer l when step t's forward pass runs.  The cache starts clean; at
    t == W every layer in P = {l >= L} is overwritten in place and never
    restored.  W = 0 (onset before any decoding step) overwrites before the
    loop.
    """
    cache = ["C"] * N
    patched = [l for l in range(N) if l >= L]
    if W == 0:
        for l in patched:
            cache[l] = "D"
    state = {}
    for t in range(1, T + 1):
        if t == W:
            for l in patched:
                cache[l] = "D"
        for l in range(N):
            state[(l, t)] = cache[l]
    return state


def sdpa_reference(shp: Shape, inputs, cell: Cell, l: int, t: int, span: str):
    """torch fp64 SDPA over an explicitly built cache (span 'C', 'D' or 'Z')."""
    f = lambda u: torch.from_numpy(so.bf16_to_f64(u))
    ck, cv = inputs.clean_kv(cell.prompt, l)
    if span == "C":
        pk, pv = f(ck), f(cv)
    elif span == "Z":
        pk, pv = torch.zeros(f(ck).shape, dtype=torch.float64), torch.zeros(f(cv).shape, dtype=torch.float64)
    else:
        dk, dv = inputs.donor_kv(cell.prompt, cell.slot, l)
        pk, pv = f(dk), f(dv)
    sk, sv = inputs.suffix_kv(0, l, 0, t)
    K = torch.cat([pk, f(sk)], dim=1)
    V = torch.cat([pv, f(sv)], dim=1)
    G = shp.num_q_heads // shp.num_kv_heads
    K = K.repeat_interleave(G, dim=0)
    V = V.repeat_interleave(G, dim=0)
    q = f(inputs.q(0, t, l))[:, None, :]
    n = K.shape[1]
    qpos = shp.prompt_len + t - 1
    mask = torch.ones(1, n, dtype=torch.bool)
    is_global = shp.sliding_window <= 0 or (shp.global_every > 0 and (l + 1) % shp.global_every == 0)
    if not is_global:
        pos = torch.arange(n)
        mask = ((qpos - pos) < shp.sliding_window)[None, :]
    if n == 0 or not bool(mask.any()):
        return np.zeros((shp.num_q_heads, shp.head_dim))
    out = torch.nn.functional.scaled_dot_product_attention(q, K, V, attn_mask=mask, scale=shp.sm_scale)
    return out[:, 0, :].numpy()


# --------------------------------------------------------------------------
# splice rule
# --------------------------------------------------------------------------
def test_splice_rule_matches_hand_table():
    rows = 0
    with open(os.path.join(GOLDEN, "splice_rule_tiny.txt")) as fh:
        for line in fh:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            head, tail = line.split(":")
            L, W, l = map(int, head.split())
            want = tail.split()
            for t, w in enumerate(want, start=1):
                src = oracle.splice_source(L, W, 0, WL.BLANK, l, t)
                got = "D" if src == so.SRC_DONOR0 else "C"
                assert got == w, (L, W, l, t)
                rows += 1
    assert rows == 60 * 4


@pytest.mark.parametrize("N,T", [(1, 1), (3, 4), (6, 9), (4, 17)])
def test_splice_rule_matches_literal_algorithm1(N, T):
    for L in range(0, N + 2):
        for W in range(0, T + 3):
            state = alg1_span_by_layer(N, T, L, W)
            for (l, t), s in state.items():
                for kind, want_d in ((WL.BLANK, so.SRC_DONOR0 + 3), (WL.ZERO, so.SRC_ZERO)):
                    got = oracle.splice_source(L, W, 3, kind, l, t)
                    assert got == (want_d if s == "D" else so.SRC_CLEAN), (L, W, l, t, kind)


def test_splice_rule_monotone_in_layer_and_step():
    for L in range(0, 7):
        for W in range(0, 9):
            for l in range(6):
                for t in range(1, 9):
                    if oracle.splice_source(L, W, 0, WL.BLANK, l, t) != so.SRC_CLEAN:
                        for l2 in range(l, 6):
                            for t2 in range(t, 9):
                                assert oracle.splice_source(L, W, 0, WL.BLANK, l2, t2) != so.SRC_CLEAN


# --------------------------------------------------------------------------
# hand-derived cases
# --------------------------------------------------------------------------
def _hand_cases():
    with open(os.path.join(GOLDEN, "hand_cases.json")) as fh:
        return json.load(fh)["cases"]


def _run_hand_case(case):
    shp = Shape(case["num_layers"], case["num_q_heads"], case["num_kv_heads"],
                case["head_dim"], case["prompt_len"], case["max_steps"],
                tuple(KIND[k] for k in case["slot_kinds"]), case["sliding_window"],
                case["global_every"], math.log(2.0))
    inp = ArrayInputs(case["q"], case["clean_k"], case["clean_v"], case["donor_k"],
                      case["donor_v"], case["suffix_k"], case["suffix_v"])
    results = []
    for qd in case["queries"]:
        cell = Cell(0, qd["slot"], qd["L"], qd["W"])
        got = oracle.decode_attn(shp, inp, 0, cell, qd["l"], qd["t"])
        want = np.array([[float(Fraction(x)) for x in row] for row in qd["expected"]])
        results.append((qd, got, want))
    return results


@pytest.mark.parametrize("case", _hand_cases(), ids=lambda c: c["name"])
def test_hand_cases(case):
    for qd, got, want in _run_hand_case(case):
        np.testing.assert_allclose(got, want, rtol=0, atol=1e-12, err_msg=qd["why"])


# --------------------------------------------------------------------------
# ZERO closed form (Table 1)
# --------------------------------------------------------------------------
@pytest.mark.parametrize("window,gevery", [(0, 0), (5, 2)])
def test_zero_donor_closed_form(window, gevery):
    shp = Shape(3, 4, 2, 8, 6, 5, (WL.ZERO,), window, gevery, 0.7)
    inp = RandomInputs(shp, 1, seed=11)
    G = shp.num_q_heads // shp.num_kv_heads
    for l in range(3):
        for t in range(0, 6):
            cell = Cell(0, 0, 0, 0)
            got = oracle.decode_attn(shp, inp, 0, cell, l, t)
            # visible prompt positions and generated entries
            qpos = shp.prompt_len + t - 1
            glob = window <= 0 or (l + 1) % gevery == 0
            lo = 0 if glob else max(0, qpos - window + 1)
            n_prompt_vis = max(0, shp.prompt_len - lo)
            i_lo = max(0, lo - shp.prompt_len)
            q = so.bf16_to_f64(inp.q(0, t, l))
            sk, sv = inp.suffix_kv(0, l, 0, t)
            sk, sv = so.bf16_to_f64(sk), so.bf16_to_f64(sv)
            want = np.zeros_like(got)
            for h in range(shp.num_q_heads):
                kv = h // G
                e = np.exp(shp.sm_scale * (sk[kv, i_lo:] @ q[h]))
                den = n_prompt_vis + e.sum()
                if den > 0:
                    want[h] = (e @ sv[kv, i_lo:]) / den
            np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-13)
            if t == 0:
                assert np.all(got == 0.0)


# --------------------------------------------------------------------------
# library cross-check on explicitly built caches
# --------------------------------------------------------------------------
SHAPES = [
    Shape(3, 4, 2, 8, 6, 5, (WL.BLANK, WL.ZERO), 0, 0, 0.35),
    Shape(4, 8, 2, 16, 9, 6, (WL.SAME_ALGO, WL.ZERO, WL.DIFF_FAMILY), 0, 0, 1.0),
    Shape(4, 6, 6, 4, 7, 7, (WL.BLANK,), 0, 0, 0.5),
    Shape(6, 4, 1, 8, 8, 6, (WL.BLANK, WL.ZERO), 6, 3, 0.8),
]


@pytest.mark.parametrize("si", range(len(SHAPES)))
def test_oracle_matches_torch_sdpa_on_built_caches(si):
    shp = SHAPES[si]
    inp = RandomInputs(shp, len(shp.slot_kinds), seed=100 + si)
    for slot, kind in enumerate(shp.slot_kinds):
        for L in (0, 1, shp.num_layers - 1, shp.num_layers):
            for W in (0, 1, 2, shp.max_steps, shp.max_steps + 1):
                cell = Cell(0, slot, L, W)
                state = alg1_span_by_layer(shp.num_layers, shp.max_steps, L, W)
                for l in range(shp.num_layers):
                    for t in range(1, shp.max_steps + 1):
                        span = state[(l, t)]
                        if span == "D" and kind == WL.ZERO:
                            span = "Z"
                        want = sdpa_reference(shp, inp, cell, l, t, span)
                        got = oracle.decode_attn(shp, inp, 0, cell, l, t)
                        np.testing.assert_allclose(got, want, rtol=1e-10, atol=1e-12)


def test_oracle_on_synth_tiny_matches_torch_sdpa():
    """The real tiny sweep's inputs (sink keys, BLANK donor) through both paths."""
    wl = WL.get("tiny")
    inp = H.SynthInputs(wl)
    seqs = wl.sequences()

    class OneSeq:
        def __init__(self, s):
            self.s = s

        def q(self, s, t, l):
            return inp.q(self.s, t, l)

        def clean_kv(self, p, l):
            return inp.clean_kv(p, l)

        def donor_kv(self, p, k, l):
            return inp.donor_kv(p, k, l)

        def suffix_kv(self, s, l, i0, i1):
            return inp.suffix_kv(self.s, l, i0, i1)

    shp = Shape(wl.num_layers, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, wl.prompt_len,
                wl.max_steps, wl.slot_kinds, wl.sliding_window, wl.global_every, wl.sm_scale)
    for s in (0, 7, 21, 45, 79):
        cell = seqs[s]
        state = alg1_span_by_layer(wl.num_layers, wl.max_steps, cell.L, cell.W)
        for l in range(wl.num_layers):
            for t in (1, 4, 5, 16):
                span = state[(l, t)]
                if span == "D" and wl.slot_kinds[cell.slot] == WL.ZERO:
                    span = "Z"
                want = sdpa_reference(shp, OneSeq(s), cell, l, t, span)
                got = oracle.decode_attn(wl, inp, s, cell, l, t)
                np.testing.assert_allclose(got, want, rtol=1e-10, atol=1e-12)


# --------------------------------------------------------------------------
# W = 0 vs W = 1; donor equal to clean
# --------------------------------------------------------------------------
def test_w0_equals_w1_and_donor_equal_to_clean():
    shp = Shape(3, 4, 2, 8, 6, 5, (WL.BLANK,), 0, 0, 0.6)
    inp = RandomInputs(shp, 1, seed=5)
    for l in range(3):
        for t in range(1, 6):
            a = oracle.decode_attn(shp, inp, 0, Cell(0, 0, 0, 0), l, t)
            b = oracle.decode_attn(shp, inp, 0, Cell(0, 0, 0, 1), l, t)
            assert np.array_equal(a, b)
    inp.DK[0] = inp.CK
    inp.DV[0] = inp.CV
    for l in range(3):
        for t in range(1, 6):
            a = oracle.decode_attn(shp, inp, 0, Cell(0, 0, 0, 0), l, t)
            b = oracle.decode_attn(shp, inp, 0, Cell(0, 0, shp.num_layers, 0), l, t)
            assert np.array_equal(a, b)


# --------------------------------------------------------------------------
# LSE merge
# --------------------------------------------------------------------------
def test_merge_equals_single_pass_softmax():
    rng = np.random.default_rng(3)
    for trial in range(40):
        n = int(rng.integers(1, 60))
        d = int(rng.integers(1, 9))
        q = rng.normal(0, 1, d)
        K = rng.normal(0, 3, (n, d))
        V = rng.normal(0, 1, (n, d))
        K[0] *= 10.0                       # a large, sink-like logit
        cuts = sorted(set([0, n] + list(rng.integers(0, n + 1, size=int(rng.integers(0, 5))))))
        parts = [so.partial(q, K[a:b], V[a:b], 0.9) for a, b in zip(cuts[:-1], cuts[1:])]
        parts.append(so.partial(q, K[:0], V[:0], 0.9))          # an empty part
        got = so.merge_partials(parts)
        want = so.attend(q[None, :], K[None], V[None], 0, 0.9)[0]
        np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-13)


def test_merge_with_zero_closed_form_partial():
    """A ZERO span of n keys is the partial (m = 0, l = n, o = 0)."""
    rng = np.random.default_rng(4)
    for n_zero in (1, 3, 17):
        q = rng.normal(0, 1, 4)
        K = rng.normal(0, 1, (5, 4))
        V = rng.normal(0, 1, (5, 4))
        got = so.merge_partials([(0.0, float(n_zero), np.zeros(4)), so.partial(q, K, V, 1.0)])
        Kz = np.concatenate([np.zeros((n_zero, 4)), K])
        Vz = np.concatenate([np.zeros((n_zero, 4)), V])
        want = so.attend(q[None], Kz[None], Vz[None], 0, 1.0)[0]
        np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-13)


# --------------------------------------------------------------------------
# planted mistakes: each must be caught by one of the pins above
# --------------------------------------------------------------------------
def _hand_cases_pass():
    try:
        for case in _hand_cases():
            for qd, got, want in _run_hand_case(case):
                np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)
    except AssertionError:
        return False
    return True


def test_pins_catch_planted_mistakes(monkeypatch):
    assert _hand_cases_pass()
    orig_source = so.splice_source
    orig_attend = so.attend
    orig_vis = so.visible_range

    mutants = {
        "onset_strict": lambda L, W, k, kind, l, t: orig_source(L, W + 1, k, kind, l, t),
        "cutoff_strict": lambda L, W, k, kind, l, t: orig_source(L + 1, W, k, kind, l, t),
        "zero_masked": None,
        "head_map_modulo": None,
        "window_excludes_self": None,
        "suffix_short": None,
    }

    def attend_modulo(q, K, V, lo, sm_scale):
        Hq, d = q.shape
        Hkv = K.shape[0]
        out = np.zeros((Hq, V.shape[2]))
        for h in range(Hq):
            kv = h % Hkv
            z = sm_scale * (K[kv, lo:] @ q[h])
            if z.size:
                w = np.exp(z - z.max())
                out[h] = (w @ V[kv, lo:]) / w.sum()
        return out

    def spliced_masking_zero(src, ck, cv, dk=None, dv=None):
        if src == so.SRC_ZERO:
            # treat the ZERO span as absent instead of as logit-0 entries
            shape = np.asarray(ck).shape
            return np.full(shape, -1e4), np.zeros(shape)
        return orig_spliced(src, ck, cv, dk, dv)

    orig_spliced = so.spliced_prompt_kv
    for name in mutants:
        with monkeypatch.context() as m:
            if name in ("onset_strict", "cutoff_strict"):
                m.setattr(so, "splice_source", mutants[name])
            elif name == "zero_masked":
                m.setattr(so, "spliced_prompt_kv", spliced_masking_zero)
            elif name == "head_map_modulo":
                m.setattr(so, "attend", attend_modulo)
            elif name == "window_excludes_self":
                m.setattr(so, "visible_range",
                          lambda Tp, t, l, w, g: (min(orig_vis(Tp, t, l, w, g)[0] + (0 if so.layer_is_global(l, w, g) else 1),
                                                      Tp + t), Tp + t))
            elif name == "suffix_short":
                class Short:
                    pass
                m.setattr(so, "attend", lambda q, K, V, lo, s: orig_attend(q, K[:, :-1], V[:, :-1], lo, s))
            assert not _hand_cases_pass(), f"planted mistake '{name}' went unnoticed"


# --------------------------------------------------------------------------
# delta encoding of a donor span against the clean span
# --------------------------------------------------------------------------
def test_delta_encoding_hand_case():
    # T_p = 5, d = 2; bf16 bit patterns.  Position 1 differs in K only,
    # position 3 in V only, position 4 by the sign of a zero (-0 vs +0 are
    # different bit patterns, so the position is encoded).
    one, two, three, neg0 = 0x3F80, 0x4000, 0x4040, 0x8000
    ck = np.array([[one, two], [one, one], [two, two], [three, 0], [0, one]], np.uint16)
    cv = np.array([[two, one], [two, two], [one, one], [one, one], [one, 0]], np.uint16)
    dk = ck.copy()
    dv = cv.copy()
    dk[1, 1] = three
    dv[3, 0] = three
    dk[4, 0] = neg0
    mask, rk, rv = oracle.delta_encode(ck, cv, dk, dv)
    assert mask.tolist() == [False, True, False, True, True]
    assert rk.tolist() == [[one, three], [three, 0], [neg0, one]]
    assert rv.tolist() == [[two, two], [three, one], [one, 0]]
    assert oracle.pack_mask_words(mask, 2).tolist() == [0b11010, 0]
    bits = np.zeros(64, bool)
    bits[[0, 31, 32, 63]] = True
    assert oracle.pack_mask_words(bits, 2).tolist() == [0x80000001, 0x80000001]


def test_delta_encoding_round_trip_and_merge_identity():
    rng = np.random.default_rng(9)
    for trial in range(20):
        Tp, d = int(rng.integers(1, 40)), int(rng.integers(1, 6))
        ck = to_bf16(rng.normal(0, 1, (Tp, d)))
        cv = to_bf16(rng.normal(0, 1, (Tp, d)))
        dk, dv = ck.copy(), cv.copy()
        pick = rng.random(Tp) < rng.random()
        dk[pick] = to_bf16(rng.normal(0, 1, (int(pick.sum()), d)))
        vpick = rng.random(Tp) < 0.2
        dv[vpick] = to_bf16(rng.normal(0, 2, (int(vpick.sum()), d)))
        mask, rk, rv = oracle.delta_encode(ck, cv, dk, dv)
        # lossless: the donor span comes back bit for bit
        bk, bv = oracle.delta_decode(ck, cv, mask, rk, rv)
        assert np.array_equal(bk, dk) and np.array_equal(bv, dv)
        # only differing positions are encoded
        same = ~mask
        assert np.array_equal(ck[same], dk[same]) and np.array_equal(cv[same], dv[same])
        # attention over the donor span = merge of the clean span without the
        # encoded positions and the encoded rows (step 4's identity)
        q = rng.normal(0, 1, d)
        K, V = oracle.bf16_to_f64(dk), oracle.bf16_to_f64(dv)
        want = so.attend(q[None], K[None], V[None], 0, 0.8)[0]
        got = so.merge_partials([so.partial(q, oracle.bf16_to_f64(ck[same]), oracle.bf16_to_f64(cv[same]), 0.8),
                                 so.partial(q, oracle.bf16_to_f64(rk), oracle.bf16_to_f64(rv), 0.8)])
        np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-13)


def test_delta_positions_of_the_ladder_donors():
    """On the synthetic donor-noise ladder the encoded positions are exactly
    the perturbed ones (SAME_ALGO / DIFF_ALGO) or every non-scaffold position
    (BLANK / DIFF_FAMILY), and never a scaffold position."""
    base = WL.get("qwen3-8b-ladder")
    wl = WL.Workload("ladder-small", 2, 4, 2, 64, 2, 640, base.slot_kinds, 8, (0, 2), (0, 4),
                     base.scaffold_head, base.scaffold_tail, batch=40)
    inp = H.SynthInputs(wl)
    jj = np.arange(wl.prompt_len)
    scaffold = (jj < wl.scaffold_head) | (jj >= wl.prompt_len - wl.scaffold_tail)
    for p in range(2):
        for k, kind in enumerate(wl.slot_kinds):
            if kind == WL.ZERO:
                continue
            for l in range(wl.num_layers):
                ck, cv = inp.clean_kv(p, l)
                dk, dv = inp.donor_kv(p, k, l)
                for h in range(wl.num_kv_heads):
                    mask = oracle.delta_positions(ck[h], cv[h], dk[h], dv[h])
                    assert not mask[scaffold].any()
                    if kind in (WL.SAME_ALGO, WL.DIFF_ALGO):
                        assert np.array_equal(mask, inp.perturbed(p, k, jj) & ~scaffold)
                        frac = mask.sum() / (~scaffold).sum()
                        want = 0.1 if kind == WL.SAME_ALGO else 0.5
                        assert abs(frac - want) < 0.08, (kind, frac)
                    else:
                        assert mask[~scaffold].all()


def test_delta_pins_catch_planted_mistakes(monkeypatch):
    one, two = 0x3F80, 0x4000
    ck = np.array([[one], [one]], np.uint16)
    cv = np.array([[one], [one]], np.uint16)
    dk = ck.copy()
    dv = cv.copy()
    dv[1, 0] = two
    # a K-only comparison misses position 1
    with monkeypatch.context() as m:
        m.setattr(so, "delta_positions", lambda a, b, c, e: (np.asarray(a) != np.asarray(c)).any(axis=1))
        mask, rk, rv = so.delta_encode(ck, cv, dk, dv)
        assert not np.array_equal(so.delta_decode(ck, cv, mask, rk, rv)[1], dv)
    # encoding the clean rows instead of the donor's is caught by the round trip
    mask = so.delta_positions(ck, cv, dk, dv)
    assert not np.array_equal(so.delta_decode(ck, cv, mask, ck[mask], cv[mask])[1], dv)
