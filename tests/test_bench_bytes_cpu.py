"""The bench's algorithmic-byte count, on host descriptors (no GPU): one
read of every distinct (prompt, source) span a layer-step touches, every
sequence's visible generated entries, each query once, the outputs and the
appended entries (moved by the generated-span pass in the fused call); in
delta-donor mode a reader of an encoded slot adds its prompt's
clean span (shared) and the slot's encoded rows instead of the donor span."""
from types import SimpleNamespace

import numpy as np

import bench
from paper_2605_30574_gb300 import build as B
from paper_2605_30574_gb300 import splice as S
from paper_2605_30574_gb300.sweep import model_shape
from paper_2605_30574_gb300.synth import workloads as WL


def _host_batch(wl, seqs):
    B.build()
    d = S.splice_desc_create_host(model_shape(wl), wl.num_prompts, wl.prompt_len, wl.slot_kinds,
                                  [(q.prompt, q.slot, q.L, q.W) for q in seqs], wl.max_steps)
    return SimpleNamespace(wl=wl, desc=d, seqs=seqs, B=len(seqs), p0=0)


def test_bytes_by_hand():
    # 1 layer, 2 prompts, slots (SAME_ALGO, ZERO, BLANK), 2 kv heads of 64, T_p = 100
    wl = WL.Workload("bytes", 1, 4, 2, 64, 2, 100, (WL.SAME_ALGO, WL.ZERO, WL.BLANK), 4, (0, 1), (0, 2), 4, 2,
                     batch=10 ** 6)
    seqs = [WL.Seq(0, 0, 0, 0),   # reads SAME_ALGO of prompt 0
            WL.Seq(0, 1, 0, 0),   # ZERO: no span
            WL.Seq(0, 2, 1, 0),   # L = 1 = N: clean of prompt 0
            WL.Seq(1, 0, 0, 2),   # t = 1 < W: clean of prompt 1
            WL.Seq(1, 2, 0, 0)]   # BLANK of prompt 1
    sb = _host_batch(wl, seqs)
    kv_pos = 2 * 64 * 4
    q = 4 * 64 * 2
    b = bench.algorithmic_bytes(sb, 0, 1)
    # spans: (0, SAME_ALGO), (0, clean), (1, clean), (1, BLANK); 4 readers
    assert b["prompt_span_pass"] == 4 * 100 * kv_pos
    assert b["generated_span_pass"] == 5 * 1 * kv_pos + 5 * q
    assert b["merge"] == 5 * 4 * 64 * 4 and b["append"] == 5 * 2 * 64 * 8
    # the total is the per-step formula: spans + generated entries + B Hq d (2 q + 4 out) + appends
    assert sum(b.values()) == 4 * 100 * kv_pos + 5 * 1 * kv_pos + 5 * 4 * 64 * (2 + 4) + 5 * 2 * 64 * 8
    bf = bench.algorithmic_bytes(sb, 0, 1, fused=True)
    assert bf["append"] == 0 and bf["generated_span_pass"] == b["generated_span_pass"] + b["append"]
    assert sum(bf.values()) == sum(b.values())
    # delta mode for SAME_ALGO (stored slot 0): prompt 0's reader adds the
    # clean span it already shares and 7 + 5 encoded rows (two kv heads)
    counts = np.zeros((2, 2, 1, 2), np.int64)
    counts[0, 0, 0] = (7, 5)
    counts[1, 0, 0] = (40, 40)                 # prompt 1 has no SAME_ALGO reader at this step
    bd = bench.algorithmic_bytes(sb, 0, 1, ([True, False, False], counts))
    assert bd["prompt_span_pass"] == 3 * 100 * kv_pos + (7 + 5) * 64 * 4
    assert bd["generated_span_pass"] == b["generated_span_pass"]
