"""GPU-vs-GPU invariants that the paper's definition fixes, checked bit for bit
on the CUDA path (no oracle involved):

* C1 clean equivalence (§3): a cell that is never patched (L >= N or W > T)
  gives exactly the output of a clean-only batch;
* C3 by reference == physical copy: reading donor spans through the
  descriptor equals attention over a physically spliced per-sequence cache;
* C5 W = 0 and W = 1 give the same run (reading of the onset);
* C7 permuting the batch permutes the outputs;
* the generated-span append writes exactly slot t - 1 (Algorithm 1).
"""
import numpy as np
import pytest
import torch

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


def small_wl():
    return WL.Workload("inv", 4, 8, 2, 128, 2, 300, (WL.SAME_ALGO, WL.ZERO, WL.BLANK), 12,
                       (0, 2, 4), (0, 1, 5, 13), 8, 4, batch=10 ** 6)


def test_clean_equivalence_bit_exact():
    wl = small_wl()
    seqs = wl.sequences()
    clean_seqs = [WL.Seq(q.prompt, q.slot, wl.num_layers, q.W) for q in seqs]
    a = SweepBatch(wl, seqs=seqs)
    b = SweepBatch(wl, seqs=clean_seqs)
    for t in (1, 4, 5, 12):
        for l in range(wl.num_layers):
            oa = a.run(l, t).clone()
            ob = b.run(l, t).clone()
            m = S.splice_debug_source_map(a.desc, l, t)
            same = [s for s in range(len(seqs)) if m[s] == S.SRC_CLEAN]
            diff = [s for s in range(len(seqs)) if m[s] != S.SRC_CLEAN]
            assert same
            assert torch.equal(oa[same], ob[same]), (l, t)
            if diff:
                assert not torch.equal(oa[diff], ob[diff])


def test_w0_equals_w1_bit_exact():
    wl = small_wl()
    s0 = [WL.Seq(q.prompt, q.slot, q.L, 0) for q in wl.sequences()]
    s1 = [WL.Seq(q.prompt, q.slot, q.L, 1) for q in wl.sequences()]
    a = SweepBatch(wl, seqs=s0)
    b = SweepBatch(wl, seqs=s1)
    for t in (1, 2, 12):
        for l in range(wl.num_layers):
            assert torch.equal(a.run(l, t), b.run(l, t)), (l, t)


def test_permutation_bit_exact():
    wl = small_wl()
    seqs = wl.sequences()
    a = SweepBatch(wl, seqs=seqs)
    perm = torch.randperm(len(seqs), generator=torch.Generator().manual_seed(3))
    b = SweepBatch(wl, seqs=[seqs[i] for i in perm.tolist()], fill=False)
    b.k_clean.copy_(a.k_clean)
    b.v_clean.copy_(a.v_clean)
    b.k_donor.copy_(a.k_donor)
    b.v_donor.copy_(a.v_donor)
    pc = perm.cuda()
    b.k_suffix.copy_(a.k_suffix[pc])
    b.v_suffix.copy_(a.v_suffix[pc])
    for t in (1, 5, 12):
        for l in range(wl.num_layers):
            a.gen_inputs(l, t)
            a.attn(l, t)
            b.q.copy_(a.q[pc])
            b.attn(l, t)
            assert torch.equal(b.out, a.out[pc]), (l, t)


def test_by_reference_equals_physical_copy():
    wl = small_wl()
    seqs = wl.sequences()
    a = SweepBatch(wl, seqs=seqs)
    Bn = len(seqs)
    # one "prompt" per sequence holding the span it reads, every cell clean
    phys_wl = WL.Workload("phys", wl.num_layers, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, Bn,
                          wl.prompt_len, (WL.BLANK,), wl.max_steps, (0,), (0,), 0, 0, batch=Bn)
    phys_seqs = [WL.Seq(s, 0, wl.num_layers, 0) for s in range(Bn)]
    b = SweepBatch(phys_wl, seqs=phys_seqs, fill=False)
    b.k_suffix.copy_(a.k_suffix)
    b.v_suffix.copy_(a.v_suffix)
    stored = {k: i for i, k in enumerate(k for k, kd in enumerate(wl.slot_kinds) if kd != WL.ZERO)}
    for t in (1, 5, 12):
        for l in range(wl.num_layers):
            m = S.splice_debug_source_map(a.desc, l, t)
            for s, q in enumerate(seqs):
                p = q.prompt - a.p0
                if m[s] == S.SRC_CLEAN:
                    b.k_clean[s, l].copy_(a.k_clean[p, l])
                    b.v_clean[s, l].copy_(a.v_clean[p, l])
                elif m[s] == S.SRC_ZERO:
                    b.k_clean[s, l].zero_()
                    b.v_clean[s, l].zero_()
                else:
                    st = stored[m[s] - S.SRC_DONOR0]
                    b.k_clean[s, l].copy_(a.k_donor[p, st, l])
                    b.v_clean[s, l].copy_(a.v_donor[p, st, l])
            a.gen_inputs(l, t)
            a.attn(l, t)
            b.q.copy_(a.q)
            b.attn(l, t)
            nz = [s for s in range(Bn) if m[s] != S.SRC_ZERO]
            z = [s for s in range(Bn) if m[s] == S.SRC_ZERO]
            assert torch.equal(a.out[nz], b.out[nz]), (l, t)
            if z:
                assert_close(a.out[z].cpu().numpy(), b.out[z].cpu().numpy().astype(np.float64), f"zero l={l} t={t}")


def test_append_writes_exactly_slot_t_minus_1():
    wl = small_wl()
    a = SweepBatch(wl, seqs=wl.sequences())
    g = H.SynthInputs(wl)
    before = a.k_suffix.clone()
    l, t = 2, 7
    a.k_suffix[:, l, :, t - 1].zero_()
    a.v_suffix[:, l, :, t - 1].zero_()
    a.gen_inputs(l, t)
    a.append(l, t)
    torch.cuda.synchronize()
    assert torch.equal(a.k_suffix, before)
    ks = a.k_suffix.view(torch.int16).cpu().numpy().view(np.uint16)
    vs = a.v_suffix.view(torch.int16).cpu().numpy().view(np.uint16)
    for s in (0, 5, len(a.seqs) - 1):
        k, v = g.suffix_kv(s, l, t - 1, t)
        assert np.array_equal(ks[s, l, :, t - 1], k[:, 0]) and np.array_equal(vs[s, l, :, t - 1], v[:, 0])


def test_argument_errors_on_device_descriptor():
    wl = small_wl()
    a = SweepBatch(wl, seqs=wl.sequences())
    with pytest.raises(S.SpliceError) as e:
        S.spliced_decode_attn(a.desc, 0, wl.max_steps + 1, a.q, a.k_clean, a.v_clean, a.k_donor, a.v_donor,
                              a.k_suffix, a.v_suffix, a.out, a.ws)
    assert e.value.status == S.EINVAL
    with pytest.raises(S.SpliceError) as e:
        S.spliced_decode_attn(a.desc, 0, 1, a.q, a.k_clean, a.v_clean, a.k_donor, a.v_donor,
                              a.k_suffix, a.v_suffix, a.out, a.ws, workspace_bytes=16)
    assert e.value.status == S.EINVAL
    with pytest.raises(S.SpliceError) as e:
        S.spliced_decode_attn(a.desc, 0, 1, a.q.data_ptr() + 2, a.k_clean, a.v_clean, a.k_donor, a.v_donor,
                              a.k_suffix, a.v_suffix, a.out, a.ws)
    assert e.value.status == S.EINVAL
    with pytest.raises(S.SpliceError) as e:
        S.suffix_kv_append(a.desc, 0, 0, a.k_new, a.v_new, a.k_suffix, a.v_suffix)
    assert e.value.status == S.EINVAL
    S.splice_check_device_error(a.desc)


def test_workspace_alignment_does_not_change_results():
    """The workspace need only be 16-byte aligned: the library places its
    partial-state arrays on 256-byte boundaries inside it, so an offset
    pointer gives the same bits."""
    wl = small_wl()
    a = SweepBatch(wl, seqs=wl.sequences())
    nbytes = S.splice_workspace_bytes(a.desc)
    big = torch.empty(nbytes + 256, dtype=torch.uint8, device="cuda")
    for l, t in ((0, 1), (3, 5), (1, 12)):
        ref = a.run(l, t).clone()
        for off in (16, 48, 240):
            a.out.fill_(float("nan"))
            S.spliced_decode_attn(a.desc, l, t, a.q, a.k_clean, a.v_clean, a.k_donor, a.v_donor,
                                  a.k_suffix, a.v_suffix, a.out, big.data_ptr() + off, workspace_bytes=nbytes)
            torch.cuda.synchronize()
            assert torch.equal(a.out, ref), (l, t, off)
    S.splice_check_device_error(a.desc)


def test_bounded_wait_reports_instead_of_hanging():
    """A wait that can never complete gives up after its limit and the host
    reads SPLICE_EDEVICE; the context stays usable and the record clears."""
    wl = small_wl()
    a = SweepBatch(wl, seqs=wl.sequences())
    S.splice_check_device_error(a.desc)
    S.splice_debug_wait_timeout(a.desc, 1000)          # 1 ms
    with pytest.raises(S.SpliceError) as e:
        S.splice_check_device_error(a.desc)
    assert e.value.status == S.EDEVICE
    S.splice_check_device_error(a.desc)                # cleared
    out = a.run(1, 5).clone()                           # the GPU still works
    assert torch.isfinite(out).all()
    S.splice_check_device_error(a.desc)


def test_two_descriptors_interleaved_on_one_stream():
    """Each descriptor carries its own work counters and tables: alternating
    the calls of two batches on one stream gives exactly the outputs of each
    batch's calls issued on their own."""
    wl_a = small_wl()
    wl_b = WL.Workload("inv2", 4, 8, 2, 128, 2, 300, (WL.BLANK, WL.ZERO), 12, (0, 2), (0, 3), 8, 4,
                       batch=10 ** 6, seed=5)
    a = SweepBatch(wl_a, seqs=wl_a.sequences())
    b = SweepBatch(wl_b, seqs=wl_b.sequences())
    points = [(l, t) for t in (1, 5, 12) for l in range(4)]
    alone_a = {p: a.run(*p).clone() for p in points}
    alone_b = {p: b.run(*p).clone() for p in points}
    for l, t in points:
        a.gen_inputs(l, t)
        b.gen_inputs(l, t)
        a.append(l, t)
        b.append(l, t)
        a.attn(l, t)
        b.attn(l, t)
        assert torch.equal(a.out, alone_a[(l, t)]), ("a", l, t)
        assert torch.equal(b.out, alone_b[(l, t)]), ("b", l, t)
    S.splice_check_device_error(a.desc)
    S.splice_check_device_error(b.desc)


def test_attention_reads_the_entry_appended_right_before():
    """The generated-span pass may stream its older entries while the
    append launched right before it (same layer and step) still runs; the
    entry that append writes must still be read only after it lands.  The
    slot is poisoned with large values first, so reading it early would
    swamp the softmax.  Also an append of an older slot followed by an
    attention call at a later step: the pass then waits for the append
    before it reads anything."""
    from test_gpu_parity import oracle_rows
    from parity_util import CachedInputs
    wl = WL.get("qwen3-8b-ladder")
    wl = WL.Workload("late-wait", 3, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, 2, 256, wl.slot_kinds, 64,
                     (0, 1, 3), (0, 16), wl.scaffold_head, wl.scaffold_tail, batch=10 ** 6)
    sb = SweepBatch(wl, seqs=wl.sequences())
    inp = CachedInputs(wl)
    poison = torch.tensor(40.0, dtype=torch.bfloat16)
    for l, t in ((0, 1), (1, 17), (2, 64), (1, 33)):
        sb.gen_inputs(l, t)
        torch.cuda.synchronize()
        sb.k_suffix[:, l, :, t - 1] = poison.cuda()
        sb.v_suffix[:, l, :, t - 1] = poison.cuda()
        sb.append(l, t)
        sb.attn(l, t)
        out = sb.out.cpu().numpy()
        ref = oracle_rows(wl, inp, sb.seqs, l, t, range(sb.B))
        assert_close(out, ref, f"late wait l={l} t={t}")
    # re-append an older slot, then attend a later step of the same layer
    l, t_old, t = 1, 10, 30
    sb.gen_inputs(l, t_old)
    torch.cuda.synchronize()
    sb.k_suffix[:, l, :, t_old - 1] = poison.cuda()
    sb.v_suffix[:, l, :, t_old - 1] = poison.cuda()
    sb.append(l, t_old)
    sb.gen_inputs(l, t)
    sb.attn(l, t)
    out = sb.out.cpu().numpy()
    ref = oracle_rows(wl, inp, sb.seqs, l, t, range(sb.B))
    assert_close(out, ref, f"older slot l={l} t={t}")
    S.splice_check_device_error(sb.desc)
