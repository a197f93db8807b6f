"""spliced_decode_attn_static, the entry point for callers that cannot
allocate device memory (a plugin whose host runtime owns every device
allocation, a decode loop where a synchronising cudaMalloc is not allowed).

It must give the same outputs as spliced_decode_attn with a caller-provided
workspace, call after call (the static scratch is shared and keeps the last
call's contents), and refuse descriptors whose scratch would not fit.  This
file is collected last so that a stop-at-first-failure run has already run
every other test.
"""
import os
import re

import numpy as np
import pytest
import torch

import oracle
from paper_2605_30574_gb300 import build as B
from paper_2605_30574_gb300 import splice as S
from paper_2605_30574_gb300.sweep import SweepBatch, model_shape
from paper_2605_30574_gb300.synth import workloads as WL
from parity_util import CachedInputs, assert_close

pytestmark = pytest.mark.gpu
HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "splice.h")


def _header_limit():
    with open(HEADER) as fh:
        m = re.search(r"#define\s+SPLICE_STATIC_SCRATCH_BYTES\s+\((\d+)u\s*<<\s*(\d+)\)", fh.read())
    return int(m.group(1)) << int(m.group(2))


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


def _static_call(sb, layer, step, out):
    S.spliced_decode_attn_static(sb.desc, layer, step, sb.q, sb.k_clean, sb.v_clean, sb.k_donor, sb.v_donor,
                                 sb.k_suffix, sb.v_suffix, out)


@pytest.mark.parametrize("name,points", [
    ("tiny", [(1, 5), (3, 16)]),
    ("ladder-slice", [(20, 300), (35, 17)]),
])
def test_static_scratch_matches_workspace_entry_point(name, points):
    if name == "tiny":
        wl = WL.get("tiny")
        sb = SweepBatch(wl, 0)
    else:
        base = WL.get("qwen3-8b-ladder")
        wl = WL.Workload("ladder-slice", base.num_layers, base.num_q_heads, base.num_kv_heads, base.head_dim,
                         2, 1024, base.slot_kinds, 400, base.L_values, base.W_values, base.scaffold_head,
                         base.scaffold_tail, batch=100)
        sb = SweepBatch(wl, 0)
    limit = S.splice_static_scratch_bytes()
    assert limit == _header_limit()
    assert S.splice_workspace_bytes(sb.desc) <= limit
    inp = CachedInputs(wl)
    for layer, step in points:                       # two calls in a row
        sb.gen_inputs(layer, step)
        sb.append(layer, step)
        sb.attn(layer, step)
        want = sb.out.clone()
        got = torch.full_like(sb.out, float("nan"))
        _static_call(sb, layer, step, got)
        torch.cuda.synchronize()
        # the same kernels on the same inputs, only the scratch differs
        assert torch.equal(got, want), (name, layer, step)
        # and a few rows against the fp64 oracle
        g = got.cpu().numpy()
        for s in range(0, sb.B, max(1, sb.B // 6)):
            ref = oracle.decode_attn(wl, inp, sb.s0 + s, sb.seqs[s], layer, step)
            assert_close(g[s], ref, f"{name} s={s} layer={layer} step={step}")
    S.splice_check_device_error(sb.desc)
    sb.close()


def test_static_scratch_refuses_oversized_descriptor():
    wl = WL.get("qwen3-8b-ladder")
    seqs = [(q.prompt, q.slot, q.L, q.W) for q in wl.sequences()[:2000]]
    d = S.splice_desc_create_host(model_shape(wl), wl.num_prompts, wl.prompt_len, wl.slot_kinds, seqs,
                                  wl.max_steps)
    assert S.splice_workspace_bytes(d) > S.splice_static_scratch_bytes()
    fake = 1 << 20   # never dereferenced: the size check comes first
    with pytest.raises(S.SpliceError) as e:
        S.spliced_decode_attn_static(d, 0, 1, fake, fake, fake, fake, fake, fake, fake, fake, stream=0)
    assert e.value.status == S.EINVAL
    assert "static maximum" in str(e.value)
    d.close()


def test_static_scratch_in_delta_mode():
    """The no-allocation entry point runs delta-donor mode like the
    workspace entry point (the delta buffer is the caller's, allocated once
    at setup)."""
    base = WL.get("qwen3-8b-ladder")
    wl = WL.Workload("ladder-slice-delta", 4, base.num_q_heads, base.num_kv_heads, base.head_dim, 2, 1024,
                     base.slot_kinds, 400, (0, 2, 4), base.W_values, base.scaffold_head, base.scaffold_tail,
                     batch=100)
    sb = SweepBatch(wl, 0)
    buf = torch.empty(S.splice_delta_bytes(sb.desc), dtype=torch.uint8, device="cuda")
    S.splice_delta_build(sb.desc, sb.k_clean, sb.v_clean, sb.k_donor, sb.v_donor, buf, 0.6)
    for layer, step in ((1, 20), (3, 300)):
        sb.gen_inputs(layer, step)
        sb.append(layer, step)
        sb.attn(layer, step)
        want = sb.out.clone()
        got = torch.full_like(sb.out, float("nan"))
        _static_call(sb, layer, step, got)
        torch.cuda.synchronize()
        assert torch.equal(got, want), (layer, step)
    S.splice_check_device_error(sb.desc)


def test_static_scratch_refuses_host_query():
    """The scratch is the descriptor's device's array: a q that is not device
    (or managed) memory of that device is refused before any launch."""
    wl = WL.get("tiny")
    sb = SweepBatch(wl, 0)
    q_host = torch.empty(sb.q.shape, dtype=sb.q.dtype, pin_memory=True)
    with pytest.raises(S.SpliceError) as e:
        S.spliced_decode_attn_static(sb.desc, 0, 1, q_host, sb.k_clean, sb.v_clean, sb.k_donor, sb.v_donor,
                                     sb.k_suffix, sb.v_suffix, sb.out)
    assert e.value.status == S.EINVAL
    S.splice_check_device_error(sb.desc)
    sb.close()
