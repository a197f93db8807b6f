"""The two attention passes in either order (and the order chosen per call)
give the same outputs and the same generated-span store, bit for bit: the
passes write disjoint partial states that are combined in a fixed order --
by the merge kernel, or, with the prompt-span pass first and one split of
each span, by the generated-span pass (ZERO rows at an item's end, the
others there once the prompt-span pass has completed, else at the warp's
end), in the merge kernel's operations (§3 attention over the prompt span and the generated span,
Algorithm 1's append).  Checked on a sweep where the prompt-span pass is
small (the chosen order puts it first), on the ladder-shaped sweep's full
512-sequence batch (at t = 700 the chosen order puts it second) and on head
dims 64 and 256, with sampled rows against the oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2605_30574_gb300 import build as B
from paper_2605_30574_gb300 import splice as S
from paper_2605_30574_gb300.sweep import SweepBatch
from paper_2605_30574_gb300.synth import host as H
from paper_2605_30574_gb300.synth import workloads as WL
from parity_util import assert_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


def _run_orders(sb, points):
    """{order: [(out, store slice) per point]} with every order on the same inputs."""
    got = {}
    for order in (0, 1, 2):
        S.splice_debug_pass_order(sb.desc, order)
        res = []
        for l, t in points:
            sb.gen_inputs(l, t)
            sb.step(l, t)
            res.append((sb.out.clone(), sb.k_suffix[:, l].clone(), sb.v_suffix[:, l].clone()))
        got[order] = res
    S.splice_debug_pass_order(sb.desc, 0)
    S.splice_check_device_error(sb.desc)
    return got


def _check_equal(got, points):
    for i, (l, t) in enumerate(points):
        for order in (1, 2):
            for a, b in zip(got[0][i], got[order][i]):
                assert torch.equal(a, b), (order, l, t)


def test_pass_order_small_prompt_span():
    wl = WL.get("qwen3-4b")
    sb = SweepBatch(wl, 0)
    points = [(0, 1), (5, 17), (20, 64), (35, 200)]
    got = _run_orders(sb, points)
    _check_equal(got, points)
    inp = H.SynthInputs(wl)
    l, t = points[-1]
    out = got[0][-1][0].cpu().numpy()
    for s in (0, sb.B // 3, sb.B - 1):
        ref = oracle.decode_attn(wl, inp, s, sb.seqs[s], l, t)
        assert_close(out[s], ref, f"qwen3-4b s={s} l={l} t={t}")
    sb.close()


def test_pass_order_ladder_batch():
    wl = WL.get("qwen3-8b-ladder")
    sb = SweepBatch(wl, 0)
    points = [(1, 100), (30, 700)]
    got = _run_orders(sb, points)
    _check_equal(got, points)
    inp = H.SynthInputs(wl)
    l, t = points[-1]
    out = got[0][-1][0].cpu().numpy()
    for s in (0, sb.B - 1):
        ref = oracle.decode_attn(wl, inp, s, sb.seqs[s], l, t)
        assert_close(out[s], ref, f"ladder s={s} l={l} t={t}")
    sb.close()


@pytest.mark.parametrize("name,points", [("tiny", [(0, 1), (2, 9), (3, 16)]),
                                         ("gemma3-4b", [(0, 3), (5, 100), (33, 250)])])
def test_pass_order_other_head_dims(name, points):
    wl = WL.get(name)
    sb = SweepBatch(wl, 0)
    got = _run_orders(sb, points)
    _check_equal(got, points)
    inp = H.SynthInputs(wl)
    l, t = points[-1]
    out = got[1][-1][0].cpu().numpy()
    for s in (0, sb.B // 2, sb.B - 1):
        ref = oracle.decode_attn(wl, inp, s, sb.seqs[s], l, t)
        assert_close(out[s], ref, f"{name} s={s} l={l} t={t}")
    sb.close()


def test_prompt_span_first_launches_no_merge():
    """With the prompt-span pass first and one split of each span, the
    generated-span pass merges every row and the call launches two kernels;
    with the generated-span pass first the merge kernel is launched too.
    The outputs are the same bits either way (checked above)."""
    wl = WL.get("qwen3-4b")
    sb = SweepBatch(wl, 0)
    l, t = 5, 40
    sb.gen_inputs(l, t)
    counts = {}
    for order in (1, 2):
        S.splice_debug_pass_order(sb.desc, order)
        before = S.splice_kernel_launches(sb.desc)
        sb.step(l, t)
        torch.cuda.synchronize()
        counts[order] = S.splice_kernel_launches(sb.desc) - before
    S.splice_debug_pass_order(sb.desc, 0)
    S.splice_check_device_error(sb.desc)
    assert counts == {1: 2, 2: 3}, counts
    sb.close()


def test_pass_order_rejects_bad_value():
    wl = WL.get("tiny")
    sb = SweepBatch(wl, 0)
    with pytest.raises(RuntimeError):
        S.splice_debug_pass_order(sb.desc, 3)
    sb.close()
