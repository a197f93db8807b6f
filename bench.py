#!/usr/bin/env python3
"""Benchmark of spliced decode attention on the Qwen3-8B-shaped donor-noise
ladder sweep (36 layers, 32 q / 8 kv heads, d = 128, 32 prompts x 4096-token
prompt span, 5 donor slots, 1024 decode steps, (L, W) grid 5 x 4, 512-sequence
decode batches).

One *step* = one decode step of one 512-sequence batch through all layers:
per layer one ``spliced_decode_step`` (the step's append done inside the
generated-span pass, then the attention; ``--unfused``: ``suffix_kv_append``
+ ``spliced_decode_attn``).  Steps walk the decode steps t of the sweep in a
stratified order (t_k at the midpoints of K equal slices of 1..T), so the mix
of generated-span lengths and splice epochs matches the whole run.  The
metric is sequence-steps per second (one sequence-step = all layers and heads
of one sequence at one t).

Legs (one JSON line on rank 0):
* value: device-resident inputs, CUDA events around exactly K steps;
* roofline: per-kernel launch durations from CUDA events recorded by the
  library around each launch, over a second pass of the same K steps;
  algorithmic bytes per launch from the descriptor's source maps;
* e2e: the same K steps through the C ABI with the step's queries and new
  K/V copied from pinned host memory and the outputs copied back, copies
  overlapped with compute on separate streams;
* graph: each timed step's calls (every layer) captured once into a CUDA
  graph before the timed region, then the K graphs replayed under the same
  events -- the fused-step launch mode;
* delta: the same K steps in delta-donor mode (donor spans that share most
  positions with the clean span encoded against it once, before timing);
* workloads: the Qwen3-4B-, Llama-3-8B- and Gemma-3-4B-shaped sweeps (batch
  0, fewer steps), each with its own algorithmic bytes and kernel split;
* cpu_baseline: the fp64 CPU oracle on a bounded sample of (sequence,
  layer, step) units of the same batch, on the host's cores.
``--impl reference`` times that oracle alone as the reference arm.
``--profile-case`` runs one small, fixed launch sequence for profilers (see
``profile_case``) instead of the bench.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "spliced decode-attn sequence-steps/s (Qwen3-8B-shaped sweep); HBM GB/s vs peak"
UNIT = "seq-steps/s"
WORKLOAD = "qwen3-8b-ladder"
NOMINAL_HBM_GBS = 8000.0
# DRAM bytes per algorithmic byte of a kernel, from one ncu capture of the
# reduced ladder case (read + written bytes / algorithmic bytes of that launch);
# traffic grows in proportion to the units a launch processes.  Only kernels
# whose current build was captured are listed.
TRAFFIC_PER_ALGORITHMIC_BYTE = {"generated_span_pass": (539.052 + 5.846) / 541.065,
                                "prompt_span_pass": (237.009 + 4.820) / 234.881}


def step_schedule(T: int, n: int, offset: int = 0):
    """Decode steps at the midpoints of n equal slices of 1..T."""
    return [1 + ((2 * ((k + offset) % n) + 1) * T) // (2 * n) for k in range(n)]


def rank_batch(num_batches: int, base: int, rank: int) -> int:
    """Weak scaling: rank r of the job runs sweep batch (base + r) mod #batches."""
    return (base + rank) % num_batches


def reduce_timing(ms: float, units: int, dist=None, device=None):
    """Whole-job timing: the slowest rank's time and the units of all ranks."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return ms, units
    import torch
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    u = torch.tensor([units], dtype=torch.float64, device=device)
    dist.all_reduce(u)
    return float(t.item()), int(u.item())


def read_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as fh:
            d = json.load(fh)
        return float(d.get("hbm_gbs", 6800.0)), "measured"
    return 6800.0, "fallback"


# --------------------------------------------------------------------------
# algorithmic bytes (what the method must move), from the source maps
# --------------------------------------------------------------------------
def algorithmic_bytes(sb, layer: int, step: int, delta=None, fused=False):
    """Bytes per kernel kind at (layer, step) (``fused``: the step's append
    runs inside the generated-span pass).  ``delta`` = (slot flags,
    encoded counts [prompts][stored slots][N][Hkv]) in delta mode: a reader
    of an encoded slot reads its prompt's clean span (shared with the clean
    readers) and the slot's encoded rows instead of the donor span."""
    from paper_2605_30574_gb300 import splice as S
    wl = sb.wl
    st = S.splice_plan_stats(sb.desc, layer, step)
    m = S.splice_debug_source_map(sb.desc, layer, step)
    kv_pos = wl.num_kv_heads * wl.head_dim * 4          # K + V bf16 of one position, all kv heads
    spans, rows = set(), 0
    for s, code in enumerate(m):
        if code == S.SRC_ZERO:
            continue
        p = sb.seqs[s].prompt
        if delta is not None and code >= S.SRC_DONOR0 and delta[0][code - S.SRC_DONOR0]:
            spans.add((p, S.SRC_CLEAN))
            spans.add((p, -int(code)))                  # the slot's encoded rows, counted below
        else:
            spans.add((p, code))
    for p, code in spans:
        if code < 0:
            k = -code - S.SRC_DONOR0
            stq = sum(1 for j in range(k) if wl.slot_kinds[j] != 0)
            rows += int(delta[1][p - sb.p0, stq, layer].sum()) * wl.head_dim * 4
    n_span = sum(1 for _, code in spans if code >= 0)
    q_bytes = wl.num_q_heads * wl.head_dim * 2
    append = sb.B * wl.num_kv_heads * wl.head_dim * 8 if step >= 1 else 0
    # each sequence's q counted once (with the generated-span pass, which
    # reads every sequence's q); in the fused call the append's bytes are
    # moved by the generated-span pass
    return {
        "prompt_span_pass": n_span * st["prompt_visible"] * kv_pos + rows,
        "generated_span_pass": sb.B * st["suffix_visible"] * kv_pos + sb.B * q_bytes + (append if fused else 0),
        "merge": sb.B * wl.num_q_heads * wl.head_dim * 4,
        "append": 0 if fused else append,
    }


# --------------------------------------------------------------------------
# clocks during the timed region
# --------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.fh.close()

    def summary(self):
        if not self.path or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"]}
        rows = []
        with open(self.path) as fh:
            for line in fh:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        pw = [float(r[3]) for r in rows if r[3].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        loaded = [x for x in sm if x > 0.5 * max(sm)] if sm else []
        return {"sm_mhz": statistics.median(loaded) if loaded else None,
                "sm_max_mhz": max(mx) if mx else None,
                "power_w_max": max(pw) if pw else None,
                "samples": len(rows), "reasons": reasons}


# --------------------------------------------------------------------------
# CPU oracle leg
# --------------------------------------------------------------------------
class _Provider:
    """Pre-generated oracle inputs of one (sequence, layer, step) unit."""

    def __init__(self, d):
        self.d = d

    def q(self, s, t, l):
        return self.d["q"]

    def clean_kv(self, p, l):
        return self.d["clean"]

    def donor_kv(self, p, k, l):
        return self.d["donor"]

    def suffix_kv(self, s, l, i0, i1):
        return self.d["suffix"]


def _make_unit_inputs(wl, s, l, t):
    import oracle
    from paper_2605_30574_gb300.synth import host as H
    g = H.SynthInputs(wl)
    seq = wl.sequences()[s]
    src = oracle.splice_source(seq.L, seq.W, seq.slot, wl.slot_kinds[seq.slot], l, t)
    d = {"q": g.q(s, t, l), "clean": g.clean_kv(seq.prompt, l), "suffix": g.suffix_kv(s, l, 0, t)}
    d["donor"] = g.donor_kv(seq.prompt, seq.slot, l) if src >= oracle.SRC_DONOR0 else None
    return seq, d


def _oracle_worker(name, units, barrier, results):
    import oracle
    from paper_2605_30574_gb300.synth import workloads as W
    wl = W.get(name)
    prepared = [(s, l, t) + _make_unit_inputs(wl, s, l, t) for (s, l, t) in units]
    barrier.wait()
    t0 = time.perf_counter()
    for s, l, t, seq, d in prepared:
        oracle.decode_attn(wl, _Provider(d), s, seq, l, t)
    results.put((len(prepared), time.perf_counter() - t0))


def plan_units(wl, batch, seed):
    """(s, l, t) units of the parity sampling plan inside one sweep batch,
    shuffled: every cell of the batch's first and last prompts at steps {1,
    W - 1, W, W + 1, T / 2, T} of the cell's own onset, every layer."""
    lo, hi = wl.batch_range(batch)
    seqs = wl.sequences()
    N, T = wl.num_layers, wl.max_steps
    ends = {seqs[lo].prompt, seqs[hi - 1].prompt}
    units = []
    for s in range(lo, hi):
        q = seqs[s]
        if q.prompt not in ends:
            continue
        steps = sorted({x for x in (1, q.W - 1, q.W, q.W + 1, T // 2, T) if 1 <= x <= T})
        units += [(s, l, t) for l in range(N) for t in steps]
    rng = np.random.default_rng(seed)
    rng.shuffle(units)
    return units


def run_oracle_sample(name, per_core):
    """Times the oracle on per_core[c] units in process c (generation excluded);
    returns (units, wall seconds of the slowest process)."""
    import multiprocessing as mp
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[k] = "1"
    ctx = mp.get_context("spawn")
    barrier = ctx.Barrier(len(per_core) + 1)
    results = ctx.Queue()
    procs = [ctx.Process(target=_oracle_worker, args=(name, units, barrier, results)) for units in per_core]
    for p in procs:
        p.start()
    barrier.wait()
    t0 = time.perf_counter()
    got = [results.get() for _ in procs]
    wall = time.perf_counter() - t0
    for p in procs:
        p.join()
    return sum(g[0] for g in got), wall


def host_cores():
    """(cores the oracle uses = the CPUs this process may run on, os.cpu_count())."""
    try:
        aff = len(os.sched_getaffinity(0))
    except AttributeError:      # pragma: no cover
        aff = os.cpu_count() or 1
    return max(1, aff), os.cpu_count() or 1


def cpu_baseline(name, budget_s=8.0, batch=0):
    """The oracle on all affined cores, each process about budget_s of its
    one-thread work (so 10-30 s of CPU work in all), plus the one-thread rate."""
    from paper_2605_30574_gb300.synth import workloads as W
    wl = W.get(name)
    cores, n_cpu = host_cores()
    units = plan_units(wl, batch, seed=7)
    # one thread: 32 units alone
    n1, w1 = run_oracle_sample(name, [units[:32]])
    per_unit = w1 / max(n1, 1)
    upc = int(max(1, min(2048, budget_s / per_unit)))
    need = cores * upc
    take = (units * (need // len(units) + 1))[:need]
    n, wall = run_oracle_sample(name, [take[c::cores] for c in range(cores)])
    value = n / wall / wl.num_layers
    return {"value": value, "unit": UNIT, "cores": cores, "os_cpu_count": n_cpu, "affinity_cores": cores,
            "value_1thread": 1.0 / per_unit / wl.num_layers, "kind": "oracle",
            "sample": (f"{n} (sequence, layer, step) units of batch {batch} from the parity sampling plan (every "
                       f"cell of the batch's first and last prompts at steps 1, W-1, W, W+1, T/2, T of its own "
                       f"onset, every layer; {upc} per core), fp64 numpy oracle, input generation excluded; "
                       f"{wall:.1f} s wall on {cores} processes; seq-steps = units / {wl.num_layers} layers; "
                       f"value_1thread from {n1} units on one core"),
            "note": ("a plain per-head fp64 numpy loop, deliberately slow: the GPU/CPU ratio says nothing about "
                     "kernel quality (the roofline fraction does)")}


def reference_arm(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    from paper_2605_30574_gb300.synth import workloads as W
    wl = W.get(args.workload)
    cores, n_cpu = host_cores()
    units = plan_units(wl, args.batch, seed=11)
    per_step = [units[(k * cores + c) % len(units)] for k in range(args.warmup + args.steps) for c in range(cores)]
    for w in range(args.warmup):
        run_oracle_sample(args.workload, [[u] for u in per_step[w * cores:(w + 1) * cores]])
    total_units, total_wall = 0, 0.0
    for k in range(args.warmup, args.warmup + args.steps):
        n, wall = run_oracle_sample(args.workload, [[u] for u in per_step[k * cores:(k + 1) * cores]])
        total_units += n
        total_wall += wall
    value = total_units / total_wall / wl.num_layers
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * total_wall / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": workload_config(wl, args.batch, args.gpus),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "os_cpu_count": n_cpu, "kind": "oracle",
                             "sample": f"each step: {cores} (sequence, layer, step) units of batch {args.batch} "
                                       f"from the parity sampling plan, one per core; input generation excluded"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def workload_config(wl, batch: int, world: int) -> dict:
    """The `config` of both arms' lines: the workload, its batch, the layout
    over GPUs (identical for the same workload, whatever runs it)."""
    lo, hi = wl.batch_range(batch)
    return {"workload": describe(wl), "batch": f"batch {batch} of {wl.num_batches()}: sequences {lo}-{hi - 1}",
            "parallelism": f"{world} GPU(s), one sweep batch each, no collective"}


def describe(wl):
    return (f"{wl.name}: {wl.num_layers} layers, {wl.num_q_heads}/{wl.num_kv_heads} heads, d {wl.head_dim}, "
            f"{wl.num_prompts} prompts x {wl.prompt_len}-token span, {len(wl.slot_kinds)} donor slots, "
            f"T {wl.max_steps}, L {list(wl.L_values)} x W {list(wl.W_values)}, {wl.batch}-sequence batches")


# --------------------------------------------------------------------------
# GPU arm
# --------------------------------------------------------------------------
def make_run_step(sb, fused: bool):
    """One decode step of the whole batch through every layer, on a stream."""
    from paper_2605_30574_gb300 import splice as S
    N = sb.wl.num_layers

    def run_step(t, q, k_new, v_new, out, st):
        for l in range(N):
            if fused:
                S.spliced_decode_step(sb.desc, l, t, q[l], k_new[l], v_new[l], sb.k_clean, sb.v_clean, sb.k_donor,
                                      sb.v_donor, sb.k_suffix, sb.v_suffix, out[l], sb.ws, stream=st)
            else:
                S.suffix_kv_append(sb.desc, l, t, k_new[l], v_new[l], sb.k_suffix, sb.v_suffix, st)
                S.spliced_decode_attn(sb.desc, l, t, q[l], sb.k_clean, sb.v_clean, sb.k_donor, sb.v_donor,
                                      sb.k_suffix, sb.v_suffix, out[l], sb.ws, stream=st)
    return run_step


def gen_step_inputs(sb, ts, dev):
    """Queries and new K/V of every layer of steps ts, generated ahead (excluded from timing)."""
    import torch
    from paper_2605_30574_gb300.synth import device as SD
    wl, N = sb.wl, sb.wl.num_layers
    qs = torch.empty((len(ts), N) + tuple(sb.q.shape), dtype=torch.bfloat16, device=dev)
    kn = torch.empty((len(ts), N) + tuple(sb.k_new.shape), dtype=torch.bfloat16, device=dev)
    vn = torch.empty_like(kn)
    for i, t in enumerate(ts):
        for l in range(N):
            SD.fill_q(wl, sb.s0, l, t, qs[i, l])
            SD.fill_new_kv(wl, sb.s0, l, t, kn[i, l], vn[i, l])
    return qs, kn, vn


def profile_pass(sb, steps, qs, kn, vn, outs, run_step, stream):
    """The same steps with the library's per-launch events: {kind: (launches, ms)}."""
    import torch
    from paper_2605_30574_gb300 import splice as S
    S.splice_profile_enable(sb.desc, True)
    S.splice_profile_read(sb.desc)
    torch.cuda.synchronize()
    for i, t in enumerate(steps):
        run_step(t, qs[i], kn[i], vn[i], outs, stream)
    torch.cuda.synchronize()
    prof = S.splice_profile_read(sb.desc)
    S.splice_profile_enable(sb.desc, False)
    return prof


def kernel_table(prof, per_kind):
    """Per kernel kind: launches, summed time, share of the serialised step,
    algorithmic GB/s, algorithmic bytes per launch and -- where an ncu capture
    gave the kernel's DRAM bytes per algorithmic byte -- DRAM bytes per launch."""
    total = sum(x[1] for x in prof.values()) or 1.0
    out = {}
    for k, v in prof.items():
        per_launch = per_kind[k] // max(v[0], 1)
        ratio = TRAFFIC_PER_ALGORITHMIC_BYTE.get(k)
        out[k] = {"launches": v[0], "ms_total": round(v[1], 3), "share": round(v[1] / total, 4),
                  "GBps": round(per_kind[k] / (v[1] / 1000.0) / 1e9, 1) if v[1] > 0 else None,
                  "bytes_per_launch": per_launch,
                  "traffic_per_launch": round(ratio * per_launch) if ratio and v[0] else None}
    return out


def step_bytes(sb, steps, fused):
    per_kind = {"append": 0, "prompt_span_pass": 0, "generated_span_pass": 0, "merge": 0}
    for t in steps:
        for l in range(sb.wl.num_layers):
            for k, v in algorithmic_bytes(sb, l, t, fused=fused).items():
                per_kind[k] += v
    return per_kind


def gpu_arm(args):
    import torch
    import torch.distributed as dist
    from paper_2605_30574_gb300 import build as B
    from paper_2605_30574_gb300 import splice as S
    from paper_2605_30574_gb300.sweep import SweepBatch
    from paper_2605_30574_gb300.synth import workloads as W

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    B.build()
    fused = not args.unfused
    wl = W.get(args.workload)
    batch = rank_batch(wl.num_batches(), args.batch, rank)
    sb = SweepBatch(wl, batch)
    N = wl.num_layers
    steps = step_schedule(wl.max_steps, args.steps)
    warm = step_schedule(wl.max_steps, max(args.warmup, 1), offset=0)[: args.warmup]
    dev = torch.device("cuda", local)
    qs, kn, vn = gen_step_inputs(sb, steps, dev)
    wq, wkn, wvn = gen_step_inputs(sb, warm, dev) if warm else (None, None, None)
    outs = torch.empty((N,) + tuple(sb.out.shape), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()
    run_step = make_run_step(sb, fused)

    for i, t in enumerate(warm):
        run_step(t, wq[i], wkn[i], wvn[i], outs, stream)
    torch.cuda.synchronize()

    # ---- value: exactly K steps, device-resident inputs ----
    launches0 = S.splice_kernel_launches(sb.desc)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        ev0.record(stream)
        for i, t in enumerate(steps):
            run_step(t, qs[i], kn[i], vn[i], outs, stream)
        ev1.record(stream)
        torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    ms = ev0.elapsed_time(ev1)
    gpu_launches = S.splice_kernel_launches(sb.desc) - launches0
    S.splice_check_device_error(sb.desc)

    units = sb.B * len(steps)
    ms, units = reduce_timing(ms, units, dist if world > 1 else None, dev)
    value = units / (ms / 1000.0)

    # ---- algorithmic bytes of the timed steps, and the roofline pass ----
    per_kind = step_bytes(sb, steps, fused)
    total_bytes = sum(per_kind.values())
    prof = profile_pass(sb, steps, qs, kn, vn, outs, run_step, stream)
    peak, peak_kind = read_peaks()
    dom = max(prof, key=lambda k: prof[k][1])
    n_l, ms_l = prof[dom]
    achieved = (per_kind[dom] / max(n_l, 1)) / ((ms_l / max(n_l, 1)) / 1000.0) / 1e9
    kernels = kernel_table(prof, per_kind)

    # ---- graph: every timed step captured once, then replayed ----
    graph = None
    if not args.no_graph:
        graph = graph_leg(sb, steps, qs, kn, vn, outs, run_step, world, dist)

    # ---- delta: donor spans encoded against the clean spans ----
    delta = None
    if not args.no_delta and sb.Dst:
        delta = delta_leg(sb, steps, qs, kn, vn, outs, run_step, world, dist, per_kind, fused)

    # ---- e2e: host buffers through the C ABI, copies overlapped ----
    e2e = None
    if not args.no_e2e:
        e2e = e2e_leg(sb, steps, qs, kn, vn, run_step, dev)
    del qs, kn, vn, wq, wkn, wvn, outs
    sb.close()
    del sb
    torch.cuda.empty_cache()

    # ---- the other model-shaped sweeps ----
    workloads = None
    if not args.no_workloads and rank == 0 and world == 1:
        workloads = {name: workload_leg(name, args.workload_steps, fused, dev, peak)
                     for name in ("qwen3-4b", "llama3-8b", "gemma3-4b") if name != args.workload}

    if rank == 0:
        cpu = None if args.no_cpu_baseline else cpu_baseline(args.workload, batch=batch)
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": len(steps),
            "warmup": args.warmup, "ms_per_step": ms / len(steps), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": workload_config(wl, batch, world),
            "call": "spliced_decode_step (append fused into the generated-span pass)" if fused
                    else "suffix_kv_append + spliced_decode_attn",
            "decode_steps_t": steps, "l2": "inputs larger than L2 (every step streams >10 GB); no flush",
            "hbm": {"algorithmic_GB_per_step": round(total_bytes / len(steps) / 1e9, 3),
                    "achieved_GBps": round(total_bytes / (ms / 1000.0) / 1e9, 1),
                    "frac_of_measured": round(total_bytes / (ms / 1000.0) / 1e9 / peak, 4),
                    "frac_of_8TBps": round(total_bytes / (ms / 1000.0) / 1e9 / NOMINAL_HBM_GBS, 4)},
            "roofline": {"kernel": dom, "bound": "hbm", "achieved": round(achieved, 1), "peak": peak,
                         "unit": "GB/s", "frac": round(achieved / peak, 4), "peak_source": peak_kind,
                         "traffic": (round(TRAFFIC_PER_ALGORITHMIC_BYTE[dom] * per_kind[dom] / max(n_l, 1))
                                     if dom in TRAFFIC_PER_ALGORITHMIC_BYTE else None),
                         "bytes_per_launch": per_kind[dom] // max(n_l, 1),
                         "ms_per_launch": ms_l / max(n_l, 1)},
            "kernels": kernels,
            "e2e": e2e, "graph": graph, "delta": delta, "workloads": workloads, "gpu_launches": gpu_launches,
            "clocks": clk.summary(), "cpu_baseline": cpu,
        }
        print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()
    return 0


def workload_leg(name, n_steps, fused, dev, peak, warmup=2):
    """One of the other model-shaped sweeps: batch 0, n_steps stratified
    steps (the same timing rules), its algorithmic bytes and kernel split."""
    import torch
    from paper_2605_30574_gb300 import splice as S
    from paper_2605_30574_gb300.sweep import SweepBatch
    from paper_2605_30574_gb300.synth import workloads as W
    wl = W.get(name)
    sb = SweepBatch(wl, 0)
    steps = step_schedule(wl.max_steps, n_steps)
    warm = step_schedule(wl.max_steps, warmup)
    qs, kn, vn = gen_step_inputs(sb, steps, dev)
    wq, wkn, wvn = gen_step_inputs(sb, warm, dev)
    outs = torch.empty((wl.num_layers,) + tuple(sb.out.shape), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()
    run_step = make_run_step(sb, fused)
    for i, t in enumerate(warm):
        run_step(t, wq[i], wkn[i], wvn[i], outs, stream)
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(dev.index or 0) as clk:
        ev0.record(stream)
        for i, t in enumerate(steps):
            run_step(t, qs[i], kn[i], vn[i], outs, stream)
        ev1.record(stream)
        torch.cuda.synchronize()
    ms = ev0.elapsed_time(ev1)
    S.splice_check_device_error(sb.desc)
    per_kind = step_bytes(sb, steps, fused)
    total = sum(per_kind.values())
    prof = profile_pass(sb, steps, qs, kn, vn, outs, run_step, stream)
    ideal = peak * 1e9 / (total / len(steps)) * sb.B
    value = sb.B * len(steps) / (ms / 1000.0)
    out = {"workload": describe(wl), "batch": f"batch 0: {sb.B} sequences", "steps": len(steps),
           "decode_steps_t": steps, "value": value, "unit": UNIT, "ms_per_step": ms / len(steps),
           "algorithmic_GB_per_step": round(total / len(steps) / 1e9, 3),
           "achieved_GBps": round(total / (ms / 1000.0) / 1e9, 1),
           "frac_of_measured": round(total / (ms / 1000.0) / 1e9 / peak, 4),
           "ideal_seq_steps_per_s_at_measured_peak": round(ideal, 1),
           "kernels": kernel_table(prof, per_kind), "clocks": clk.summary()}
    del qs, kn, vn, wq, wkn, wvn, outs
    sb.close()
    del sb
    torch.cuda.empty_cache()
    return out


def graph_leg(sb, steps, qs, kn, vn, outs, run_step, world, dist):
    """The K timed steps, each captured into one CUDA graph (all layers'
    append + attention) outside the timed region and replayed inside it."""
    import torch
    from paper_2605_30574_gb300 import splice as S
    graphs = []
    for i, t in enumerate(steps):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            run_step(t, qs[i], kn[i], vn[i], outs, torch.cuda.current_stream())
        graphs.append(g)
    for g in graphs[:3]:
        g.replay()
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    ev0.record()
    for g in graphs:
        g.replay()
    ev1.record()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    ms = ev0.elapsed_time(ev1)
    S.splice_check_device_error(sb.desc)
    units = sb.B * len(steps)
    ms, units = reduce_timing(ms, units, dist if world > 1 else None, torch.device("cuda", torch.cuda.current_device()))
    del graphs
    return {"value": units / (ms / 1000.0), "unit": UNIT, "ms_per_step": ms / len(steps),
            "how": "each timed step (all layers: append + attention) captured once into a CUDA graph before "
                   "the timed region; the K graphs replayed under CUDA events"}


def delta_leg(sb, steps, qs, kn, vn, outs, run_step, world, dist, plain_bytes, fused, max_fraction=0.6):
    """The K timed steps in delta-donor mode: the batch's stored donor spans
    encoded against the clean spans once, before the timed region (slots
    whose encoded fraction is at most max_fraction), then the same steps
    timed under CUDA events; the prompt-span pass timed per launch after."""
    import torch
    from paper_2605_30574_gb300 import splice as S
    wl, N = sb.wl, sb.wl.num_layers
    buf = torch.empty(S.splice_delta_bytes(sb.desc), dtype=torch.uint8, device=sb.k_clean.device)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    frac = S.splice_delta_build(sb.desc, sb.k_clean, sb.v_clean, sb.k_donor, sb.v_donor, buf, max_fraction)
    build_s = time.perf_counter() - t0
    flags = [f >= 0 and f <= max_fraction for f in frac]
    # encoded counts, from the buffer's count part
    spans = sb.Pl * sb.Dst * N * wl.num_kv_heads
    w32 = 4 * ((wl.prompt_len + 127) // 128)
    count_off = (spans * w32 * 4 + 255) // 256 * 256
    counts = buf[count_off: count_off + spans * 4].view(torch.int32).cpu().numpy().reshape(
        sb.Pl, sb.Dst, N, wl.num_kv_heads)
    stream = torch.cuda.current_stream()
    for i, t in enumerate(steps[:2]):
        run_step(t, qs[i], kn[i], vn[i], outs, stream)
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    ev0.record(stream)
    for i, t in enumerate(steps):
        run_step(t, qs[i], kn[i], vn[i], outs, stream)
    ev1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    ms = ev0.elapsed_time(ev1)
    S.splice_check_device_error(sb.desc)
    per_kind = {"append": 0, "prompt_span_pass": 0, "generated_span_pass": 0, "merge": 0}
    for t in steps:
        for l in range(N):
            for k, v in algorithmic_bytes(sb, l, t, (flags, counts), fused=fused).items():
                per_kind[k] += v
    prof = profile_pass(sb, steps, qs, kn, vn, outs, run_step, stream)
    S.splice_delta_clear(sb.desc)
    del buf
    units = sb.B * len(steps)
    ms, units = reduce_timing(ms, units, dist if world > 1 else None, torch.device("cuda", torch.cuda.current_device()))
    pp = prof["prompt_span_pass"]
    return {"value": units / (ms / 1000.0), "unit": UNIT, "ms_per_step": ms / len(steps),
            "slot_fraction": [round(f, 4) for f in frac], "slots_encoded": [int(f) for f in flags],
            "encode_s": round(build_s, 3),
            "prompt_span_algorithmic_GB_per_step": round(per_kind["prompt_span_pass"] / len(steps) / 1e9, 3),
            "prompt_span_algorithmic_GB_per_step_plain": round(plain_bytes["prompt_span_pass"] / len(steps) / 1e9, 3),
            "prompt_span_pass_ms_per_step": round(pp[1] / len(steps), 3),
            "prompt_span_pass_GBps": round(per_kind["prompt_span_pass"] / (pp[1] / 1000.0) / 1e9, 1) if pp[1] else None,
            "how": f"stored donor slots with at most {max_fraction:.0%} of their positions differing from the clean "
                   "span encoded once before the timed region (splice_delta_build); readers of an encoded slot "
                   "read the clean span with those positions masked plus the encoded rows; same K steps"}


def e2e_leg(sb, steps, qs, kn, vn, run_step, dev):
    import torch
    K = len(steps)
    N = sb.wl.num_layers
    h_q = torch.empty(qs.shape, dtype=qs.dtype, pin_memory=True)
    h_kn = torch.empty(kn.shape, dtype=kn.dtype, pin_memory=True)
    h_vn = torch.empty(vn.shape, dtype=vn.dtype, pin_memory=True)
    h_q.copy_(qs.cpu())
    h_kn.copy_(kn.cpu())
    h_vn.copy_(vn.cpu())
    # three device slots for inputs and outputs: a copy over the host link
    # has two compute steps to finish before its slot is needed again
    NB = 3
    d_q = [torch.empty(qs.shape[1:], dtype=qs.dtype, device=dev) for _ in range(NB)]
    d_kn = [torch.empty(kn.shape[1:], dtype=kn.dtype, device=dev) for _ in range(NB)]
    d_vn = [torch.empty(vn.shape[1:], dtype=vn.dtype, device=dev) for _ in range(NB)]
    d_out = [torch.empty((N,) + tuple(sb.out.shape), dtype=torch.float32, device=dev) for _ in range(NB)]
    h_out = [torch.empty((N,) + tuple(sb.out.shape), dtype=torch.float32, pin_memory=True) for _ in range(NB)]
    comp = torch.cuda.current_stream()
    h2d = torch.cuda.Stream()
    d2h = torch.cuda.Stream()

    def pipeline():
        in_ready = [torch.cuda.Event() for _ in range(K)]
        comp_done = [torch.cuda.Event() for _ in range(K)]
        out_free = [torch.cuda.Event() for _ in range(K)]
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(h2d)
        for k, t in enumerate(steps):
            b = k % NB
            with torch.cuda.stream(h2d):
                if k >= NB:
                    h2d.wait_event(comp_done[k - NB])         # slot b no longer read by compute
                d_q[b].copy_(h_q[k], non_blocking=True)
                d_kn[b].copy_(h_kn[k], non_blocking=True)
                d_vn[b].copy_(h_vn[k], non_blocking=True)
                in_ready[k].record(h2d)
            comp.wait_event(in_ready[k])
            if k >= NB:
                comp.wait_event(out_free[k - NB])             # output slot b copied out
            run_step(t, d_q[b], d_kn[b], d_vn[b], d_out[b], comp)
            comp_done[k].record(comp)
            with torch.cuda.stream(d2h):
                d2h.wait_event(comp_done[k])
                h_out[b].copy_(d_out[b], non_blocking=True)
                out_free[k].record(d2h)
        e1.record(d2h)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1)

    pipeline()          # untimed: first-use costs of the copy path
    ms = pipeline()
    h2d_bytes = (qs[0].numel() + kn[0].numel() + vn[0].numel()) * 2
    d2h_bytes = d_out[0].numel() * 4
    return {"value": sb.B * K / (ms / 1000.0), "unit": UNIT, "h2d_bytes_per_step": int(h2d_bytes),
            "d2h_bytes_per_step": int(d2h_bytes), "ms_per_step": ms / K,
            "how": "pinned host queries + new K/V per step copied H2D, outputs of every layer copied D2H, "
                   "on two copy streams overlapped with compute (three device slots)"}


def profile_case(args):
    """A small, fixed launch sequence for profilers: one decode step of a
    reduced copy of a sweep (same heads, head dim, prompt span, donor slots
    and (L, W) grid shape, but few layers, a shorter generated-span store and
    a smaller batch) so a capture holds a few GB on the device while every
    launch still streams more than the 129 MB L2.  Repeated --reps times."""
    import torch
    from paper_2605_30574_gb300 import build as B
    from paper_2605_30574_gb300 import splice as S
    from paper_2605_30574_gb300.sweep import SweepBatch
    from paper_2605_30574_gb300.synth import workloads as W
    B.build()
    base = W.get(args.workload)
    layers = args.layers
    Ls = tuple(sorted({min(layers, round(L * layers / base.num_layers)) for L in base.L_values}))
    wl = W.Workload(base.name + "-prof", layers, base.num_q_heads, base.num_kv_heads, base.head_dim,
                    base.num_prompts, base.prompt_len, base.slot_kinds, args.step + 8, Ls, base.W_values,
                    base.scaffold_head, base.scaffold_tail, batch=args.batch_size,
                    sliding_window=base.sliding_window, global_every=base.global_every, sm_scale=base.sm_scale)
    sb = SweepBatch(wl, 0)
    # algorithmic bytes of every launch of one repetition, for comparing a
    # capture's DRAM counters with what the launch must move
    for l in range(wl.num_layers):
        ab = algorithmic_bytes(sb, l, args.step, fused=not args.unfused)
        print(f"layer {l}: algorithmic bytes per launch " +
              ", ".join(f"{k} {v}" for k, v in ab.items() if v))
    for _ in range(args.reps):
        for l in range(wl.num_layers):
            sb.gen_inputs(l, args.step)
            if args.unfused:
                sb.append(l, args.step)
                sb.attn(l, args.step)
            else:
                sb.step(l, args.step)
    torch.cuda.synchronize()
    S.splice_check_device_error(sb.desc)
    gb = (sb.k_suffix.numel() + sb.k_clean.numel() + (sb.k_donor.numel() if sb.k_donor is not None else 0)) * 4 / 1e9
    print(f"profile case ok: {wl.name}, {sb.B} sequences, step {args.step}, {wl.num_layers} layers, "
          f"{args.reps} reps, stores {gb:.2f} GB, {'unfused' if args.unfused else 'fused'} calls")
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=16)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=WORKLOAD)
    ap.add_argument("--batch", type=int, default=0)
    ap.add_argument("--unfused", action="store_true", help="suffix_kv_append + spliced_decode_attn per layer")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-graph", action="store_true")
    ap.add_argument("--no-delta", action="store_true")
    ap.add_argument("--no-workloads", action="store_true")
    ap.add_argument("--workload-steps", type=int, default=8, help="timed steps of each other sweep")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--profile-case", action="store_true", help="run the small profiling case instead")
    ap.add_argument("--layers", type=int, default=4, help="profile case: layers")
    ap.add_argument("--batch-size", type=int, default=256, help="profile case: sequences")
    ap.add_argument("--step", type=int, default=512, help="profile case: decode step")
    ap.add_argument("--reps", type=int, default=3, help="profile case: repetitions")
    args = ap.parse_args(argv)
    if args.profile_case:
        return profile_case(args)
    if args.impl == "reference":
        return reference_arm(args)
    return gpu_arm(args)


if __name__ == "__main__":
    sys.exit(main())
