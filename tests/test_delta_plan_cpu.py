"""Delta-mode planning on the host (no GPU).

In delta mode a reader of an encoded donor slot is stacked into its prompt's
clean-span tiles with a row mask (its stored slot + 1) and also reads the
slot's encoded rows in tiles of their own; everything else is planned as
before.  Checked row by row against the splice rule's source map, for the
donor-noise ladder's encodable slots and for every stored slot of the small
sweeps.
"""
import collections

import pytest

from paper_2605_30574_gb300 import build as B
from paper_2605_30574_gb300 import splice as S
from paper_2605_30574_gb300.sweep import model_shape
from paper_2605_30574_gb300.synth import workloads as WL


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


def _host_desc(wl, seqs):
    return S.splice_desc_create_host(model_shape(wl), wl.num_prompts, wl.prompt_len, wl.slot_kinds,
                                     [(q.prompt, q.slot, q.L, q.W) for q in seqs], wl.max_steps)


def _stored_index(kinds):
    out, n = {}, 0
    for k, kind in enumerate(kinds):
        if kind != WL.ZERO:
            out[k] = n
            n += 1
    return out


def _check_table(wl, seqs, d, flags, l, t):
    kinds = wl.slot_kinds
    stored = _stored_index(kinds)
    G = wl.num_q_heads // wl.num_kv_heads
    per_tile = max(1, 128 // G)
    m = S.splice_debug_source_map(d, l, t)
    rows = S.splice_debug_plan_rows(d, l, t)
    by_seq = collections.defaultdict(list)
    tiles = collections.defaultdict(list)
    for tile, src, s, mask in rows:
        by_seq[s].append((src, mask))
        tiles[tile].append((src, s, mask))
    for s, code in enumerate(m):
        got = sorted(by_seq.get(s, []))
        if code == S.SRC_ZERO:
            assert got == [], (s, got)
        elif code == S.SRC_CLEAN:
            assert got == [(S.SRC_CLEAN, 0)], (s, got)
        else:
            k = code - S.SRC_DONOR0
            if flags[k]:
                assert got == sorted([(S.SRC_CLEAN, stored[k] + 1), (S.GROUP_DELTA | code, 0)]), (s, got)
            else:
                assert got == [(code, 0)], (s, got)
    # every tile holds one group source and one prompt; span tiles first,
    # delta tiles after them; masked rows after the unmasked ones of a tile
    seen_delta = False
    order = sorted(tiles)
    assert order == list(range(len(order)))
    for tile in order:
        rs = tiles[tile]
        srcs = {src for src, _, _ in rs}
        assert len(srcs) == 1 and len(rs) <= per_tile
        assert len({seqs[s].prompt for _, s, _ in rs}) == 1
        is_delta = next(iter(srcs)) & S.GROUP_DELTA != 0
        if is_delta:
            seen_delta = True
        else:
            assert not seen_delta, "a span tile after a delta tile"
        masks = [mask for _, _, mask in rs]
        assert masks == sorted(masks)
    st = S.splice_plan_stats(d, l, t)
    assert st["num_tiles"] == len(order)


@pytest.mark.parametrize("flags", [(1, 1, 0, 0, 0), (1, 1, 1, 1, 0), (0, 0, 0, 0, 0), (0, 1, 0, 1, 0)])
def test_ladder_delta_plan(flags):
    wl = WL.get("qwen3-8b-ladder")
    seqs = wl.sequences()[: wl.batch]
    d = _host_desc(wl, seqs)
    S.splice_debug_plan_delta(d, flags)
    for l in (0, 9, 20, 35):
        for t in (0, 1, 16, 100, 300, wl.max_steps):
            _check_table(wl, seqs, d, flags, l, t)


@pytest.mark.parametrize("name", ["tiny", "qwen3-4b"])
def test_small_sweeps_delta_plan(name):
    wl = WL.get(name)
    seqs = wl.sequences()[: wl.batch]
    d = _host_desc(wl, seqs)
    flags = [1 if k != WL.ZERO else 0 for k in wl.slot_kinds]
    S.splice_debug_plan_delta(d, flags)
    for l in range(0, wl.num_layers, max(1, wl.num_layers // 4)):
        for t in (0, 1, 4, wl.max_steps):
            _check_table(wl, seqs, d, flags, l, t)


def test_delta_flags_off_restore_the_plan():
    wl = WL.get("qwen3-8b-ladder")
    seqs = wl.sequences()[: wl.batch]
    d = _host_desc(wl, seqs)
    before = {(l, t): S.splice_debug_plan_rows(d, l, t) for l in (0, 20) for t in (1, 300)}
    S.splice_debug_plan_delta(d, (1, 1, 1, 1, 0))
    assert S.splice_debug_plan_rows(d, 20, 300) != before[(20, 300)]
    S.splice_debug_plan_delta(d, (0, 0, 0, 0, 0))
    for k, v in before.items():
        assert S.splice_debug_plan_rows(d, *k) == v


def test_delta_calls_refuse_host_descriptors_and_bad_arguments():
    wl = WL.get("tiny")
    seqs = wl.sequences()[:8]
    d = _host_desc(wl, seqs)
    assert S.splice_delta_bytes(d) > 0
    with pytest.raises(S.SpliceError) as ei:
        S.splice_delta_build(d, 16, 16, 16, 16, 16, 1.0, delta_bytes=1 << 30, stream=0)
    assert ei.value.status == S.ESTATE
    with pytest.raises(S.SpliceError) as ei:
        S.splice_delta_clear(d, stream=0)
    assert ei.value.status == S.ESTATE
    # delta-buffer layout: mask words, counts, then K and V rows of every span
    N, Hkv, Tp, dd = wl.num_layers, wl.num_kv_heads, wl.prompt_len, wl.head_dim
    spans = wl.num_prompts * 1 * N * Hkv
    w32 = 4 * ((Tp + 127) // 128)
    al = lambda x: (x + 255) // 256 * 256
    k_off = al(al(spans * w32 * 4) + spans * 4)
    rows = spans * Tp * dd * 2
    assert S.splice_delta_bytes(d) == al(k_off + rows) + rows
