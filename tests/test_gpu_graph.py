"""A whole decode step -- every layer's generated-span append and spliced
attention -- captured into one CUDA graph and replayed.

The library's calls must be capture-safe (no synchronisation, no
allocation; the programmatic dependent launch between the two attention
passes becomes a graph edge), and a replayed step must give exactly the
outputs of the same calls issued one by one, replay after replay (the
prompt-span pass's work counter is reset by its last CTA inside the graph).
"""
import pytest
import torch

from paper_2605_30574_gb300 import build as B
from paper_2605_30574_gb300.sweep import SweepBatch
from paper_2605_30574_gb300.synth import workloads as WL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


def ladder_slice(layers=6):
    base = WL.get("qwen3-8b-ladder")
    Ls = (0, 2, 4, layers)
    return WL.Workload("ladder-graph", layers, base.num_q_heads, base.num_kv_heads, base.head_dim, 2, 1024,
                       base.slot_kinds, 400, Ls, base.W_values, base.scaffold_head, base.scaffold_tail, batch=100)


@pytest.mark.parametrize("step", [17, 300])
def test_decode_step_graph_replays_bit_exact(step):
    wl = ladder_slice()
    sb = SweepBatch(wl, 0)
    N = wl.num_layers
    qs, kns, vns = [], [], []
    for l in range(N):
        sb.gen_inputs(l, step)
        qs.append(sb.q.clone())
        kns.append(sb.k_new.clone())
        vns.append(sb.v_new.clone())
    outs_eager = [torch.empty_like(sb.out) for _ in range(N)]
    for l in range(N):
        sb.append(l, step, kns[l], vns[l])
        sb.attn(l, step, q=qs[l], out=outs_eager[l])
    torch.cuda.synchronize()

    outs_graph = [torch.full_like(sb.out, float("nan")) for _ in range(N)]
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for l in range(N):
            sb.append(l, step, kns[l], vns[l])
            sb.attn(l, step, q=qs[l], out=outs_graph[l])
    for _ in range(2):
        for o in outs_graph:
            o.fill_(float("nan"))
        g.replay()
        torch.cuda.synchronize()
        for l in range(N):
            assert torch.equal(outs_graph[l], outs_eager[l]), f"layer {l}"
    # and the replayed step against the fp64 oracle on sampled rows of every layer
    import oracle
    from parity_util import CachedInputs, assert_close
    inp = CachedInputs(wl)
    for l in range(N):
        g_l = outs_graph[l].cpu().numpy()
        for s in range(0, sb.B, 9):
            ref = oracle.decode_attn(wl, inp, sb.s0 + s, sb.seqs[s], l, step)
            assert_close(g_l[s], ref, f"graph layer {l} s={s} step={step}")
    from paper_2605_30574_gb300 import splice as S
    S.splice_check_device_error(sb.desc)
    sb.close()


def test_decode_step_graph_in_delta_mode():
    """Delta-donor mode captures and replays like the default mode: the
    replayed step equals the same calls issued one by one, replay after
    replay, and both are within the path's tolerance of the fp64 oracle on
    sampled rows (the oracle reads the donor spans themselves)."""
    import numpy as np
    import oracle
    from parity_util import CachedInputs, assert_close
    from paper_2605_30574_gb300 import splice as S
    wl = ladder_slice(layers=4)
    sb = SweepBatch(wl, 0)
    buf = torch.empty(S.splice_delta_bytes(sb.desc), dtype=torch.uint8, device="cuda")
    frac = S.splice_delta_build(sb.desc, sb.k_clean, sb.v_clean, sb.k_donor, sb.v_donor, buf, 0.6)
    assert sum(1 for f in frac if 0 <= f <= 0.6) == 2        # SAME_ALGO and DIFF_ALGO
    step, N = 300, wl.num_layers
    qs, kns, vns = [], [], []
    for l in range(N):
        sb.gen_inputs(l, step)
        qs.append(sb.q.clone())
        kns.append(sb.k_new.clone())
        vns.append(sb.v_new.clone())
    outs_eager = [torch.empty_like(sb.out) for _ in range(N)]
    for l in range(N):
        sb.append(l, step, kns[l], vns[l])
        sb.attn(l, step, q=qs[l], out=outs_eager[l])
    torch.cuda.synchronize()
    outs_graph = [torch.full_like(sb.out, float("nan")) for _ in range(N)]
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for l in range(N):
            sb.append(l, step, kns[l], vns[l])
            sb.attn(l, step, q=qs[l], out=outs_graph[l])
    for _ in range(2):
        for o in outs_graph:
            o.fill_(float("nan"))
        g.replay()
        torch.cuda.synchronize()
        for l in range(N):
            assert torch.equal(outs_graph[l], outs_eager[l]), f"layer {l}"
    inp = CachedInputs(wl)
    rows = list(range(0, sb.B, 7))
    for l in (0, N - 1):
        ref = np.stack([oracle.decode_attn(wl, inp, s, sb.seqs[s], l, step) for s in rows])
        assert_close(outs_graph[l][torch.tensor(rows, device="cuda")].cpu().numpy(), ref, f"delta graph l={l}")
    S.splice_check_device_error(sb.desc)
    sb.close()


def test_fused_decode_step_graph_replays_bit_exact():
    """A whole decode step through the fused call (every layer's append done
    inside its generated-span pass) captured into one graph: replays equal
    the unfused calls issued one by one, outputs and generated-span store."""
    wl = ladder_slice()
    a = SweepBatch(wl, 0)
    b = SweepBatch(wl, 0)
    N, step = wl.num_layers, 300
    qs, kns, vns = [], [], []
    for l in range(N):
        a.gen_inputs(l, step)
        qs.append(a.q.clone())
        kns.append(a.k_new.clone())
        vns.append(a.v_new.clone())
    outs_eager = [torch.empty_like(a.out) for _ in range(N)]
    for l in range(N):
        a.append(l, step, kns[l], vns[l])
        a.attn(l, step, q=qs[l], out=outs_eager[l])
    torch.cuda.synchronize()
    outs_graph = [torch.full_like(b.out, float("nan")) for _ in range(N)]
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for l in range(N):
            b.step(l, step, q=qs[l], k_new=kns[l], v_new=vns[l], out=outs_graph[l])
    for _ in range(2):
        for o in outs_graph:
            o.fill_(float("nan"))
        b.k_suffix[:, :, :, step - 1].zero_()
        b.v_suffix[:, :, :, step - 1].zero_()
        g.replay()
        torch.cuda.synchronize()
        for l in range(N):
            assert torch.equal(outs_graph[l], outs_eager[l]), f"layer {l}"
        assert torch.equal(b.k_suffix, a.k_suffix) and torch.equal(b.v_suffix, a.v_suffix)
    from paper_2605_30574_gb300 import splice as S
    S.splice_check_device_error(b.desc)
    a.close()
    b.close()
