"""Device twin of the input generator is bit-identical to the host twin."""
import numpy as np
import pytest
import torch

from paper_2605_30574_gb300 import build as B
from paper_2605_30574_gb300.synth import device as SD
from paper_2605_30574_gb300.synth import host as H
from paper_2605_30574_gb300.synth import workloads as WL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


def u16(t):
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


@pytest.mark.parametrize("seed,stream,idx0,n,mult", [
    (0, 1, 0, 4096, 1.0), (3, 7, 123456789, 10000, 20.0), (11, 2, (1 << 40) + 5, 777, 0.088388346),
])
def test_normal_stream_bit_exact(seed, stream, idx0, n, mult):
    out = torch.empty(n, dtype=torch.int16, device="cuda")
    SD.normal(seed, stream, idx0, n, mult, out)
    torch.cuda.synchronize()
    want = H.normal_bf16(seed, stream, np.arange(idx0, idx0 + n, dtype=np.uint64), np.float32(mult))
    assert np.array_equal(u16(out), want)


def test_tiny_stores_bit_exact():
    wl = WL.get("tiny")
    g = H.SynthInputs(wl)
    N, Hkv, Tp, d, T = wl.num_layers, wl.num_kv_heads, wl.prompt_len, wl.head_dim, wl.max_steps
    kc = torch.empty((2, N, Hkv, Tp, d), dtype=torch.int16, device="cuda")
    vc = torch.empty_like(kc)
    SD.fill_clean(wl, 0, kc, vc)
    kd = torch.empty((2, 1, N, Hkv, Tp, d), dtype=torch.int16, device="cuda")
    vd = torch.empty_like(kd)
    SD.fill_donor(wl, 0, kd, vd)
    ks = torch.empty((80, N, Hkv, T, d), dtype=torch.int16, device="cuda")
    vs = torch.empty_like(ks)
    SD.fill_suffix(wl, 0, ks, vs)
    torch.cuda.synchronize()
    kc, vc, kd, vd, ks, vs = map(u16, (kc, vc, kd, vd, ks, vs))
    for p in range(2):
        for l in range(N):
            a, b = g.clean_kv(p, l)
            assert np.array_equal(kc[p, l], a) and np.array_equal(vc[p, l], b)
            a, b = g.donor_kv(p, 0, l)
            assert np.array_equal(kd[p, 0, l], a) and np.array_equal(vd[p, 0, l], b)
    for s in (0, 17, 79):
        for l in range(N):
            a, b = g.suffix_kv(s, l, 0, T)
            assert np.array_equal(ks[s, l], a) and np.array_equal(vs[s, l], b)


def test_ladder_donors_and_step_inputs_bit_exact():
    wl = WL.get("qwen3-8b-ladder")
    g = H.SynthInputs(wl)
    N, Hkv, Hq, Tp, d = wl.num_layers, wl.num_kv_heads, wl.num_q_heads, wl.prompt_len, wl.head_dim
    kd = torch.empty((1, 4, N, Hkv, Tp, d), dtype=torch.int16, device="cuda")
    vd = torch.empty_like(kd)
    SD.fill_donor(wl, 5, kd, vd)                       # prompt 5, the four stored slots
    torch.cuda.synchronize()
    kd, vd = u16(kd), u16(vd)
    for st, slot in enumerate((0, 1, 2, 3)):
        for l in (0, 20):
            a, b = g.donor_kv(5, slot, l, 0, 600)
            assert np.array_equal(kd[0, st, l, :, :600], a) and np.array_equal(vd[0, st, l, :, :600], b)
    q = torch.empty((7, Hq, d), dtype=torch.int16, device="cuda")
    kn = torch.empty((7, Hkv, d), dtype=torch.int16, device="cuda")
    vn = torch.empty_like(kn)
    SD.fill_q(wl, 1000, 9, 300, q)
    SD.fill_new_kv(wl, 1000, 9, 300, kn, vn)
    torch.cuda.synchronize()
    for i in range(7):
        assert np.array_equal(u16(q)[i], g.q(1000 + i, 300, 9))
        a, b = g.suffix_kv(1000 + i, 9, 299, 300)
        assert np.array_equal(u16(kn)[i], a[:, 0]) and np.array_equal(u16(vn)[i], b[:, 0])
