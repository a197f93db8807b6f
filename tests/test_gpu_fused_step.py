"""spliced_decode_step: one layer of one decode step with the step's append
done inside the generated-span pass (Algorithm 1's loop body: the forward
pass appends the step's generated K/V, then the step attends over the prompt
span and its generated entries, §3).

* Outputs and the generated-span store afterwards are bit-identical to
  suffix_kv_append followed by spliced_decode_attn on the same inputs, at
  every (head dim, rows per item) the generated-span pass is built for, on
  sliding-window layers, and with the step's own entry alone in its 16-key
  block, last in it, or in the middle of one.
* Launch ordering: every kernel of the library waits for the work queued
  before it on the stream before it reads its inputs.  A producer kernel
  that lets its dependents launch at once but writes q (or the new K/V) only
  after a delay must not change any output, for the fused and the unfused
  call.
"""
import pytest
import torch

from paper_2605_30574_gb300 import build as B
from paper_2605_30574_gb300 import splice as S
from paper_2605_30574_gb300.sweep import SweepBatch
from paper_2605_30574_gb300.synth import workloads as WL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


SHAPES = [
    # name, N, Hq, Hkv, d, P, Tp, kinds, T, window, global_every
    ("g4_d64", 2, 8, 2, 64, 2, 130, (WL.BLANK, WL.ZERO), 40, 0, 0),
    ("g8_d128_two_row_chunks", 2, 16, 2, 128, 1, 97, (WL.DIFF_ALGO, WL.ZERO), 40, 0, 0),
    ("g2_d256_window", 3, 4, 2, 256, 1, 200, (WL.BLANK, WL.ZERO), 40, 150, 3),
    ("g1_d128", 2, 4, 4, 128, 1, 60, (WL.SAME_ALGO,), 40, 0, 0),
    ("g6_d64", 2, 12, 2, 64, 1, 33, (WL.DIFF_FAMILY, WL.ZERO), 40, 0, 0),
]


def _wl(spec):
    name, N, Hq, Hkv, d, P, Tp, kinds, T, win, gev = spec
    Ls = tuple(sorted({0, 1, N}))
    Ws = tuple(sorted({0, 3, 17, T + 1}))
    return WL.Workload(name, N, Hq, Hkv, d, P, Tp, kinds, T, Ls, Ws, min(4, Tp), min(2, Tp), batch=10 ** 6,
                       sliding_window=win, global_every=gev)


@pytest.mark.parametrize("spec", SHAPES, ids=lambda e: e[0])
def test_fused_step_bit_identical_to_append_then_attn(spec):
    wl = _wl(spec)
    a = SweepBatch(wl, 0)
    b = SweepBatch(wl, 0)
    # entry t - 1 alone in its block (t = 1, 17, 33), last in it (16, 32), in the middle (9, 40 - 1)
    for t in (1, 9, 16, 17, 32, 33, 39, 40):
        for l in range(wl.num_layers):
            a.gen_inputs(l, t)
            b.q.copy_(a.q)
            b.k_new.copy_(a.k_new)
            b.v_new.copy_(a.v_new)
            a.append(l, t)
            a.attn(l, t)
            b.out.fill_(float("nan"))
            b.step(l, t)
            torch.cuda.synchronize()
            assert torch.equal(a.out, b.out), (spec[0], l, t)
            assert torch.equal(a.k_suffix[:, l, :, t - 1], b.k_suffix[:, l, :, t - 1]), (spec[0], l, t)
            assert torch.equal(a.v_suffix[:, l, :, t - 1], b.v_suffix[:, l, :, t - 1]), (spec[0], l, t)
    assert torch.equal(a.k_suffix, b.k_suffix) and torch.equal(a.v_suffix, b.v_suffix)
    S.splice_check_device_error(a.desc)
    S.splice_check_device_error(b.desc)


def _ladder_slice():
    base = WL.get("qwen3-8b-ladder")
    return WL.Workload("ladder-order", 4, base.num_q_heads, base.num_kv_heads, base.head_dim, 2, 1024,
                       base.slot_kinds, 400, (0, 2, 4), base.W_values, base.scaffold_head, base.scaffold_tail,
                       batch=100)


@pytest.mark.parametrize("fused", [False, True])
def test_early_signalling_producer_of_inputs(fused):
    """A producer that lets its dependents launch before it has written q
    (and, for the fused call, the new K/V) must not be overtaken."""
    wl = _ladder_slice()
    sb = SweepBatch(wl, 0)
    l, t = 3, 300
    sb.gen_inputs(l, t)
    q_true, kn_true, vn_true = sb.q.clone(), sb.k_new.clone(), sb.v_new.clone()
    # reference: the same call on inputs written long before it
    if fused:
        sb.step(l, t)
    else:
        sb.append(l, t)
        sb.attn(l, t)
    torch.cuda.synchronize()
    want = sb.out.clone()
    for _ in range(3):
        # stale inputs, then late copies of the true ones right before the call
        sb.q.zero_()
        sb.k_new.zero_()
        sb.v_new.zero_()
        sb.out.fill_(float("nan"))
        if fused:
            S.splice_debug_late_copy(sb.k_new, kn_true, 200)
            S.splice_debug_late_copy(sb.v_new, vn_true, 200)
            S.splice_debug_late_copy(sb.q, q_true, 400)        # the call's direct predecessor
            sb.step(l, t)
        else:
            S.splice_debug_late_copy(sb.q, q_true, 400)
            sb.attn(l, t)
        torch.cuda.synchronize()
        assert torch.equal(sb.out, want)
    S.splice_check_device_error(sb.desc)


def test_fused_step_rejects_step_zero_and_missing_rows():
    wl = WL.get("tiny")
    sb = SweepBatch(wl, 0)
    with pytest.raises(S.SpliceError) as e:
        sb.step(0, 0)
    assert e.value.status == S.EINVAL
    with pytest.raises(S.SpliceError) as e:
        S.spliced_decode_step(sb.desc, 0, 1, sb.q, None, sb.v_new, sb.k_clean, sb.v_clean, sb.k_donor, sb.v_donor,
                              sb.k_suffix, sb.v_suffix, sb.out, sb.ws)
    assert e.value.status == S.EINVAL
