"""Host twin of the seeded input generator: published vectors and properties."""
import numpy as np
import torch

from paper_2605_30574_gb300.synth import host as H
from paper_2605_30574_gb300.synth import workloads as WL


def test_splitmix64_published_outputs():
    # Reference outputs of Vigna's splitmix64.c: state 0 -> first output, and
    # the first five outputs from state 1234567.
    assert int(H.mix(np.array([H.GAMMA], dtype=np.uint64))[0]) == 0xE220A8397B1DCDAF
    x = np.uint64(1234567)
    with np.errstate(over="ignore"):
        outs = [int(H.mix(np.array([x + np.uint64(i + 1) * H.GAMMA], dtype=np.uint64))[0])
                for i in range(5)]
    assert outs == [6457827717110365317, 3203168211198807973, 9817491932198370423,
                    4593380528125082431, 16408922859458223821]


def test_draw_is_stream_output_i():
    x0 = H.stream_state(7, 3)
    seq = []
    x = x0
    with np.errstate(over="ignore"):
        for i in range(6):
            x = np.uint64(x + H.GAMMA)
            seq.append(int(H.mix(np.array([x], dtype=np.uint64))[0]))
    assert [int(v) for v in H.draw(7, 3, np.arange(6))] == seq


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = rng.normal(0, 3, 200000).astype(np.float32)
    # exact ties: low 16 bits == 0x8000
    ties = (rng.integers(0, 2**31, 1000, dtype=np.uint32) & np.uint32(0x7FFF0000)) | np.uint32(0x8000)
    ties = ties[(ties >> np.uint32(23)) & np.uint32(0xFF) != np.uint32(0xFF)]     # finite only
    x = np.concatenate([x, ties.view(np.float32), np.float32([0.0, -0.0, 1.0, -2.5])])
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(H.f32_to_bf16_rne(x), want)


def test_normal_constant_and_moments():
    std = np.sqrt(4 * (65536.0 ** 2 - 1) / 12)
    assert H.normal_scale() == np.float32(1.0 / std)
    z = H.normal_f32(0, 99, np.arange(1 << 20))
    assert abs(float(z.mean())) < 5e-3
    assert abs(float(z.std()) - 1.0) < 5e-3
    assert float(np.abs(z).max()) <= 131070 * float(H.normal_scale()) + 1e-6


def test_workload_tensor_scales():
    wl = WL.get("tiny")
    g = H.SynthInputs(wl)
    q = H.bf16_to_f32(g.q(3, 5, 1)).astype(np.float64)
    assert 0.5 / np.sqrt(64) < q.std() < 2.0 / np.sqrt(64)
    ck, cv = g.clean_kv(1, 2)
    ck = H.bf16_to_f32(ck).astype(np.float64)
    assert ck.shape == (2, 128, 64)
    assert 10.0 < ck[:, 0, :].std() < 30.0           # sink keys, x20
    assert 0.8 < ck[:, 1:, :].std() < 1.2
    sk, sv = g.suffix_kv(4, 1, 2, 9)
    assert sk.shape == (2, 7, 64)
    # slices agree with the full tensor
    sk_all, _ = g.suffix_kv(4, 1, 0, 16)
    assert np.array_equal(sk_all[:, 2:9], sk)


def test_donor_structure():
    wl = WL.get("qwen3-8b-ladder")
    g = H.SynthInputs(wl)
    p, l = 3, 7
    ck, cv = g.clean_kv(p, l, 0, 512)
    for k, kind in enumerate(wl.slot_kinds):
        if kind == WL.ZERO:
            continue
        dk, dv = g.donor_kv(p, k, l, 0, 512)
        # a position is "equal" if all heads and dims match
        eq = np.all(dk == ck, axis=(0, 2)) & np.all(dv == cv, axis=(0, 2))
        assert eq[:wl.scaffold_head].all()
        body = eq[wl.scaffold_head:]
        frac_eq = body.mean()
        if kind == WL.SAME_ALGO:
            assert 0.85 < frac_eq < 0.95
        elif kind == WL.DIFF_ALGO:
            assert 0.42 < frac_eq < 0.58
        else:
            assert frac_eq < 0.01
    # scaffold tail (last 12 positions)
    ckt, _ = g.clean_kv(p, l, wl.prompt_len - 12, wl.prompt_len)
    dkt, _ = g.donor_kv(p, 3, l, wl.prompt_len - 12, wl.prompt_len)   # BLANK
    assert np.array_equal(ckt, dkt)


def test_sequence_enumeration_prompt_major():
    wl = WL.get("qwen3-8b-ladder")
    seqs = wl.sequences()
    assert len(seqs) == 3200 == wl.num_sequences()
    assert seqs[0] == WL.Seq(0, 0, 0, 0)
    assert seqs[1] == WL.Seq(0, 0, 0, 16)
    assert seqs[4] == WL.Seq(0, 0, 9, 0)
    assert seqs[20] == WL.Seq(0, 1, 0, 0)
    assert seqs[100] == WL.Seq(1, 0, 0, 0)
    assert wl.num_batches() == 7
    assert wl.batch_range(6) == (3072, 3200)
    assert wl.batch_prompts(0) == (0, 6)
    for name in WL.WORKLOAD_ORDER:
        w = WL.get(name)
        assert w.num_q_heads % w.num_kv_heads == 0
    assert [WL.get(n).num_sequences() for n in WL.WORKLOAD_ORDER] == [80, 1280, 1440, 1152, 3200]
