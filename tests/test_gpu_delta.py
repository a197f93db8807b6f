"""Delta-donor mode on the GPU.

* The encoding of every stored span is bit-exact against the oracle's
  ``delta_encode``: bitmask words, counts, compacted donor rows in position
  order, and zeroed rows after them.
* Attention in delta mode matches the fp64 oracle within the path's
  tolerance: the tiny sweep exhaustively, edge shapes (ragged prompt spans,
  G = 1 / 4 / 8, d = 64 / 128 / 256, a one-position span), the ladder sweep
  at full size on sampled outputs.
* Rows of sequences that do not read a delta-encoded slot are bit-identical
  between the two modes (a row's arithmetic does not depend on its tile
  mates), and so are the readers of a donor equal to the clean span (nothing
  encoded); leaving delta mode restores the default outputs bit for bit.
* Descriptors with a sliding window are refused.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2605_30574_gb300 import build as B
from paper_2605_30574_gb300 import splice as S
from paper_2605_30574_gb300.sweep import SweepBatch
from paper_2605_30574_gb300.synth import workloads as WL
from parity_util import CachedInputs, assert_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


def delta_on(sb, max_fraction=1.0):
    buf = torch.empty(S.splice_delta_bytes(sb.desc), dtype=torch.uint8, device="cuda")
    frac = S.splice_delta_build(sb.desc, sb.k_clean, sb.v_clean, sb.k_donor, sb.v_donor, buf, max_fraction)
    return buf, frac


def layout(wl, P, Dst):
    al = lambda x: (x + 255) // 256 * 256
    spans = P * Dst * wl.num_layers * wl.num_kv_heads
    w32 = 4 * ((wl.prompt_len + 127) // 128)
    count_off = al(spans * w32 * 4)
    k_off = al(count_off + spans * 4)
    rows = spans * wl.prompt_len * wl.head_dim * 2
    return spans, w32, count_off, k_off, al(k_off + rows)


def oracle_rows(wl, inputs, seqs, l, t, which):
    return np.stack([oracle.decode_attn(wl, inputs, s, seqs[s], l, t) for s in which])


def ladder_small(d=128, Tp=700, N=3, Hq=8, Hkv=2, P=3, T=8):
    base = WL.get("qwen3-8b-ladder")
    return WL.Workload(f"ladder-delta-d{d}", N, Hq, Hkv, d, P, Tp, base.slot_kinds, T, (0, 1, N), (0, 2, T + 1),
                       base.scaffold_head, base.scaffold_tail, batch=10 ** 6)


@pytest.mark.parametrize("d", [64, 128, 256])
def test_encoding_is_bit_exact(d):
    wl = ladder_small(d=d, Tp=700 if d != 256 else 300)
    sb = SweepBatch(wl, 0)
    buf, frac = delta_on(sb)
    torch.cuda.synchronize()
    spans, w32, count_off, k_off, v_off = layout(wl, sb.Pl, sb.Dst)
    host = buf.cpu().numpy()
    words = host[: spans * w32 * 4].view(np.uint32).reshape(spans, w32)
    counts = host[count_off: count_off + spans * 4].view(np.int32)
    shape = (spans, wl.prompt_len, wl.head_dim)
    xk = host[k_off: k_off + spans * wl.prompt_len * wl.head_dim * 2].view(np.uint16).reshape(shape)
    xv = host[v_off: v_off + spans * wl.prompt_len * wl.head_dim * 2].view(np.uint16).reshape(shape)
    inp = CachedInputs(wl)
    stored = [k for k, kind in enumerate(wl.slot_kinds) if kind != WL.ZERO]
    tot = np.zeros(len(stored))
    for p in range(sb.Pl):
        for st, k in enumerate(stored):
            for l in range(wl.num_layers):
                ck, cv = inp.clean_kv(sb.p0 + p, l)
                dk, dv = inp.donor_kv(sb.p0 + p, k, l)
                for h in range(wl.num_kv_heads):
                    sp = ((p * sb.Dst + st) * wl.num_layers + l) * wl.num_kv_heads + h
                    mask, rk, rv = oracle.delta_encode(ck[h], cv[h], dk[h], dv[h])
                    n = int(mask.sum())
                    tot[st] += n
                    assert counts[sp] == n, (p, k, l, h)
                    assert np.array_equal(words[sp], oracle.pack_mask_words(mask, w32))
                    assert np.array_equal(xk[sp, :n], rk) and np.array_equal(xv[sp, :n], rv)
                    assert not xk[sp, n:].any() and not xv[sp, n:].any()
    want = tot / (sb.Pl * wl.num_layers * wl.num_kv_heads * wl.prompt_len)
    got = [frac[k] for k in stored]
    np.testing.assert_allclose(got, want, rtol=1e-6)
    assert frac[wl.slot_kinds.index(WL.ZERO)] == -1.0


def test_tiny_exhaustive_delta():
    wl = WL.get("tiny")
    sb = SweepBatch(wl, 0)
    _buf, frac = delta_on(sb)
    assert frac[0] > 0.5                 # BLANK: every non-scaffold position differs
    inp = CachedInputs(wl)
    for t in range(0, wl.max_steps + 1):
        for l in range(wl.num_layers):
            out = sb.run(l, t).cpu().numpy()
            ref = oracle_rows(wl, inp, sb.seqs, l, t, range(sb.B))
            assert_close(out, ref, f"tiny delta l={l} t={t}")
    S.splice_check_device_error(sb.desc)


EDGE = [
    # name, N, Hq, Hkv, d, P, Tp, kinds, T
    ("ragged_tp_g4_d128", 3, 8, 2, 128, 2, 300, (WL.BLANK, WL.ZERO, WL.SAME_ALGO), 9),
    ("g1_d64_tp_1", 2, 4, 4, 64, 1, 1, (WL.ZERO, WL.DIFF_FAMILY), 5),
    ("g2_d256", 3, 4, 2, 256, 2, 200, (WL.BLANK, WL.ZERO, WL.DIFF_ALGO), 12),
    ("g8_d128", 2, 16, 2, 128, 1, 129, (WL.DIFF_ALGO, WL.ZERO), 6),
    ("g3_d64_long", 2, 6, 2, 64, 1, 1100, (WL.SAME_ALGO, WL.BLANK), 300),
    # delta mode caps the span at four splits: 13000 keys are shared out evenly
    ("long_span_4_splits", 1, 4, 2, 64, 1, 13000, (WL.SAME_ALGO, WL.ZERO), 3),
]


@pytest.mark.parametrize("spec", EDGE, ids=lambda e: e[0])
def test_edge_shapes_delta(spec):
    name, N, Hq, Hkv, d, P, Tp, kinds, T = spec
    Ls = tuple(sorted({0, 1, N // 2, N}))
    Ws = tuple(sorted({0, 1, T // 2, T + 1}))
    wl = WL.Workload(name, N, Hq, Hkv, d, P, Tp, kinds, T, Ls, Ws, min(4, Tp), min(2, Tp), batch=10 ** 6)
    sb = SweepBatch(wl, 0)
    delta_on(sb)
    inp = CachedInputs(wl)
    for t in sorted({0, 1, 2, T // 2, T // 2 + 1, T}):
        for l in range(N):
            out = sb.run(l, t).cpu().numpy()
            ref = oracle_rows(wl, inp, sb.seqs, l, t, range(sb.B))
            assert_close(out, ref, f"{name} delta l={l} t={t}")
    S.splice_check_device_error(sb.desc)


def _all_outputs(sb, steps):
    outs = {}
    for t in steps:
        for l in range(sb.wl.num_layers):
            outs[(l, t)] = sb.run(l, t).clone()
    return outs


def test_modes_agree_bit_for_bit_where_nothing_is_encoded():
    wl = ladder_small(Tp=520)
    sb = SweepBatch(wl, 0)
    stored = [k for k, kind in enumerate(wl.slot_kinds) if kind != WL.ZERO]
    # make the DIFF_FAMILY donor a copy of the clean span: it encodes nothing
    k_eq = wl.slot_kinds.index(WL.DIFF_FAMILY)
    st_eq = stored.index(k_eq)
    sb.k_donor[:, st_eq].copy_(sb.k_clean)
    sb.v_donor[:, st_eq].copy_(sb.v_clean)
    steps = (1, 2, 5, 8)
    base = _all_outputs(sb, steps)
    buf, frac = delta_on(sb, max_fraction=0.6)
    assert frac[k_eq] == 0.0
    enc = {k for k in stored if frac[k] <= 0.6}
    assert enc == {wl.slot_kinds.index(WL.SAME_ALGO), wl.slot_kinds.index(WL.DIFF_ALGO), k_eq}
    inp = CachedInputs(wl)
    delta = _all_outputs(sb, steps)
    for (l, t), o in delta.items():
        m = S.splice_debug_source_map(sb.desc, l, t)
        same = [s for s in range(sb.B) if m[s] < S.SRC_DONOR0 or (m[s] - S.SRC_DONOR0) not in enc
                or (m[s] - S.SRC_DONOR0) == k_eq]
        idx = torch.tensor(same, device="cuda")
        assert torch.equal(o[idx], base[(l, t)][idx]), (l, t)
        moved = [s for s in range(sb.B) if s not in set(same)]
        if moved and t in (2, 8):
            # the oracle reads the stores as the host generator writes them;
            # the equal-to-clean copy is not among these rows
            ref = oracle_rows(wl, inp, sb.seqs, l, t, moved)
            assert_close(o[torch.tensor(moved, device="cuda")].cpu().numpy(), ref, f"delta l={l} t={t}")
    S.splice_delta_clear(sb.desc)
    again = _all_outputs(sb, steps)
    for k in base:
        assert torch.equal(again[k], base[k]), k
    S.splice_check_device_error(sb.desc)
    del buf


def test_window_descriptor_is_refused():
    wl = WL.Workload("win", 2, 4, 2, 64, 1, 64, (WL.BLANK, WL.ZERO), 8, (0, 2), (0, 4), 4, 2, batch=10 ** 6,
                     sliding_window=32, global_every=2)
    sb = SweepBatch(wl, 0)
    with pytest.raises(S.SpliceError) as ei:
        delta_on(sb)
    assert ei.value.status == S.EINVAL


def test_ladder_full_size_sampled_delta():
    from test_gpu_parity import sample_points
    wl = WL.get("qwen3-8b-ladder")
    torch.cuda.empty_cache()
    sb = SweepBatch(wl, 0)
    _buf, frac = delta_on(sb, max_fraction=0.6)
    print("ladder slot fractions", frac)
    assert frac[0] < 0.15 and 0.4 < frac[1] < 0.6 and frac[2] > 0.9 and frac[3] > 0.9
    inp = CachedInputs(wl)
    pts = sample_points(wl, sb.seqs, seed=1)
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
    del sb, _buf
    torch.cuda.empty_cache()
    worst = (0.0, 0.0)
    for (s, l, t), g in sorted(got.items(), key=lambda kv: (kv[0][1], kv[0][0])):
        ref = oracle.decode_attn(wl, inp, s, wl.sequences()[s], l, t)
        a, r = assert_close(g, ref, f"ladder delta s={s} l={l} t={t}")
        worst = (max(worst[0], a), max(worst[1], r))
    print("ladder delta points", len(got), "worst abs/rel", worst)
