"""C ABI checks that need no GPU: exported symbols, the host planner's source
map against the oracle's rule (bit-exact), plan invariants, argument
validation.  Launches are never called here except where the library must
refuse before touching CUDA."""
import ctypes
import glob
import os
import re

import numpy as np
import pytest

import oracle
from paper_2605_30574_gb300 import build as B
from paper_2605_30574_gb300 import splice as S
from paper_2605_30574_gb300.sweep import model_shape
from paper_2605_30574_gb300.synth import workloads as WL

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    B.build()
    return S.lib()


def header_functions():
    names = []
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        names += re.findall(r"^\s*(?:const\s+)?[A-Za-z_][\w]*\s*\**\s+\**(\w+)\s*\(", text, flags=re.M)
    return sorted(set(names))


def test_library_exports_every_header_function(lib):
    names = header_functions()
    assert "spliced_decode_attn" in names and "suffix_kv_append" in names and "splice_desc_create" in names
    for n in names:
        assert hasattr(lib, n), f"libsplice.so does not export {n}"
    # and the binding declares a signature for each
    assert set(names) <= set(S.SIGNATURES)


def _host_desc(wl, seqs=None):
    seqs = wl.sequences() if seqs is None else seqs
    return S.splice_desc_create_host(model_shape(wl), wl.num_prompts, wl.prompt_len, wl.slot_kinds,
                                     [(q.prompt, q.slot, q.L, q.W) for q in seqs], wl.max_steps)


def _oracle_map(wl, seqs, l, t):
    return bytes(oracle.splice_source(q.L, q.W, q.slot, wl.slot_kinds[q.slot], l, t) for q in seqs)


def test_source_map_tiny_exhaustive(lib):
    wl = WL.get("tiny")
    d = _host_desc(wl)
    seqs = wl.sequences()
    for l in range(wl.num_layers):
        for t in range(0, wl.max_steps + 1):
            assert S.splice_debug_source_map(d, l, t) == _oracle_map(wl, seqs, l, t), (l, t)


@pytest.mark.parametrize("name", ["qwen3-4b", "llama3-8b", "gemma3-4b", "qwen3-8b-ladder"])
def test_source_map_full_workloads_at_boundaries(lib, name):
    wl = WL.get(name)
    d = _host_desc(wl)
    seqs = wl.sequences()
    layers = sorted({x for L in wl.L_values for x in (L - 1, L) if 0 <= x < wl.num_layers} |
                    {0, wl.num_layers - 1})
    steps = sorted({x for W in wl.W_values for x in (W - 1, W, W + 1) if 0 <= x <= wl.max_steps} |
                   {0, 1, wl.max_steps // 2, wl.max_steps})
    for l in layers:
        for t in steps:
            assert S.splice_debug_source_map(d, l, t) == _oracle_map(wl, seqs, l, t), (l, t)


def test_source_map_arbitrary_cells_and_order(lib):
    rng = np.random.default_rng(7)
    kinds = (WL.BLANK, WL.ZERO, WL.SAME_ALGO)
    wl = WL.Workload("rand", 7, 8, 2, 64, 3, 50, kinds, 20, (0,), (0,), 4, 4, batch=1)
    seqs = [WL.Seq(int(rng.integers(0, 3)), int(rng.integers(0, 3)), int(rng.integers(0, 10)),
                   int(rng.integers(0, 25))) for _ in range(97)]
    d = _host_desc(wl, seqs)
    for l in range(7):
        for t in range(0, 21):
            assert S.splice_debug_source_map(d, l, t) == _oracle_map(wl, seqs, l, t)
    # permuting the batch permutes the map
    perm = rng.permutation(len(seqs))
    d2 = _host_desc(wl, [seqs[i] for i in perm])
    for l in (0, 3, 6):
        for t in (0, 5, 20):
            a = S.splice_debug_source_map(d, l, t)
            b = S.splice_debug_source_map(d2, l, t)
            assert bytes(a[i] for i in perm) == b


@pytest.mark.parametrize("name", ["tiny", "qwen3-8b-ladder", "gemma3-4b"])
def test_plan_groups_partition_the_readers(lib, name):
    wl = WL.get(name)
    seqs = wl.sequences()[: wl.batch]
    d = _host_desc(wl, seqs)
    G = wl.num_q_heads // wl.num_kv_heads
    per_tile = 128 // G
    for l in (0, wl.num_layers // 2, wl.num_layers - 1):
        for t in (0, 1, wl.max_steps // 3, wl.max_steps):
            m = S.splice_debug_source_map(d, l, t)
            groups = {}
            for s, code in enumerate(m):
                if code != S.SRC_ZERO:
                    groups.setdefault((seqs[s].prompt, code), []).append(s)
            st = S.splice_plan_stats(d, l, t)
            assert st["num_groups"] == len(groups)
            assert st["num_tiles"] == sum(-(-len(v) // per_tile) for v in groups.values())
            lo, hi = oracle.visible_range(wl.prompt_len, t, l, wl.sliding_window, wl.global_every)
            assert st["prompt_visible"] == max(0, wl.prompt_len - lo)
            assert st["suffix_visible"] == hi - max(lo, wl.prompt_len)


def _expect_status(fn, status):
    with pytest.raises(S.SpliceError) as ei:
        fn()
    assert ei.value.status == status, str(ei.value)


def test_argument_validation(lib):
    wl = WL.get("tiny")
    seqs = [(0, 0, 1, 2)]
    good = model_shape(wl)
    mk = lambda **kw: S.splice_desc_create_host({**good, **kw}, 2, 128, wl.slot_kinds, seqs, 16)
    _expect_status(lambda: mk(head_dim=96), S.EINVAL)
    _expect_status(lambda: mk(num_q_heads=7), S.EINVAL)
    _expect_status(lambda: mk(num_kv_heads=0), S.EINVAL)
    _expect_status(lambda: mk(num_q_heads=64, num_kv_heads=2), S.EINVAL)     # group 32 > 16
    _expect_status(lambda: mk(sm_scale=float("nan")), S.EINVAL)
    _expect_status(lambda: mk(sliding_window=-1), S.EINVAL)
    sh = good
    _expect_status(lambda: S.splice_desc_create_host(sh, 2, 128, wl.slot_kinds, [(2, 0, 0, 0)], 16), S.EINVAL)
    _expect_status(lambda: S.splice_desc_create_host(sh, 2, 128, wl.slot_kinds, [(0, 2, 0, 0)], 16), S.EINVAL)
    _expect_status(lambda: S.splice_desc_create_host(sh, 2, 128, wl.slot_kinds, [(0, 0, -1, 0)], 16), S.EINVAL)
    _expect_status(lambda: S.splice_desc_create_host(sh, 2, 128, wl.slot_kinds, [(0, 0, 0, -3)], 16), S.EINVAL)
    _expect_status(lambda: S.splice_desc_create_host(sh, 2, 128, (7,), [(0, 0, 0, 0)], 16), S.EINVAL)
    _expect_status(lambda: S.splice_desc_create_host(sh, 2, 128, (), [(0, 0, 0, 0)], 16), S.EINVAL)
    _expect_status(lambda: S.splice_desc_create_host(sh, 2, 0, wl.slot_kinds, seqs, 16), S.EINVAL)
    _expect_status(lambda: S.splice_desc_create_host(sh, 2, 128, wl.slot_kinds, seqs, 0), S.EINVAL)
    _expect_status(lambda: S.splice_desc_create_host(sh, 2, 128, wl.slot_kinds, [], 16), S.EINVAL)
    big = dict(good, num_layers=64, num_kv_heads=8, num_q_heads=8)
    _expect_status(lambda: S.splice_desc_create_host(big, 1024, 65536, wl.slot_kinds, seqs, 16), S.EINVAL)
    d = mk()
    _expect_status(lambda: S.splice_debug_source_map(d, 4, 0), S.EINVAL)
    _expect_status(lambda: S.splice_debug_source_map(d, 0, 17), S.EINVAL)
    _expect_status(lambda: S.splice_debug_source_map(d, -1, 0), S.EINVAL)
    _expect_status(lambda: S.splice_plan_stats(d, 0, -1), S.EINVAL)


def test_host_descriptor_refuses_launches(lib):
    wl = WL.get("tiny")
    d = _host_desc(wl)
    fake = 1 << 20   # never dereferenced: the call must refuse first
    _expect_status(lambda: S.spliced_decode_attn(d, 0, 1, fake, fake, fake, fake, fake, fake, fake, fake, fake,
                                                 workspace_bytes=1 << 30, stream=0), S.ESTATE)
    _expect_status(lambda: S.suffix_kv_append(d, 0, 1, fake, fake, fake, fake, stream=0), S.ESTATE)
    _expect_status(lambda: S.splice_check_device_error(d), S.ESTATE)
    assert S.splice_workspace_bytes(d) > 0
    assert S.splice_num_stored_donor_slots(d) == 1
    d.close()


def test_status_strings(lib):
    for st in range(6):
        assert S.splice_status_str(st)
    assert lib.splice_desc_destroy(None) == 0
    assert lib.splice_workspace_bytes(None) == 0


def test_pass_order_override_validated(lib):
    wl = WL.get("tiny")
    d = _host_desc(wl)
    for order in (0, 1, 2, 0):
        S.splice_debug_pass_order(d, order)
    for bad in (-1, 3):
        with pytest.raises(S.SpliceError):
            S.splice_debug_pass_order(d, bad)
