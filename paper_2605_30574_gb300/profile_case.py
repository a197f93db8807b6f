"""Small profiling case of the spliced decode-attention kernels.

Runs the launch sequence of one decode step on a reduced copy of a sweep
workload -- same heads, head dim, prompt span, donor slots and (L, W) grid
shape, but few layers, a shorter generated-span store and a smaller batch --
so that a profiler capture holds a few GB on the device while every launch
still streams more than the 129 MB L2.

    python -m paper_2605_30574_gb300.profile_case --workload qwen3-8b-ladder \\
        --layers 4 --batch 256 --step 512 --reps 3
"""
from __future__ import annotations

import argparse
import sys

import torch

from . import build as B
from . import splice as S
from .sweep import SweepBatch
from .synth import workloads as W


def reduced(wl: W.Workload, layers: int, batch: int, max_steps: int) -> W.Workload:
    # L values mapped onto the reduced depth keeps the clean / spliced mix
    Ls = tuple(sorted({min(layers, round(L * layers / wl.num_layers)) for L in wl.L_values}))
    ge = wl.global_every
    return W.Workload(wl.name + "-prof", layers, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, wl.num_prompts,
                      wl.prompt_len, wl.slot_kinds, max_steps, Ls, wl.W_values, wl.scaffold_head,
                      wl.scaffold_tail, batch=batch, sliding_window=wl.sliding_window, global_every=ge,
                      sm_scale=wl.sm_scale)


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="qwen3-8b-ladder")
    ap.add_argument("--layers", type=int, default=4)
    ap.add_argument("--batch", type=int, default=256)
    ap.add_argument("--step", type=int, default=512)
    ap.add_argument("--reps", type=int, default=3)
    args = ap.parse_args(argv)
    B.build()
    wl = reduced(W.get(args.workload), args.layers, args.batch, args.step + 8)
    sb = SweepBatch(wl, 0)
    for _ in range(args.reps):
        for l in range(wl.num_layers):
            sb.run(l, args.step)
    torch.cuda.synchronize()
    S.splice_check_device_error(sb.desc)
    gb = (sb.k_suffix.numel() + sb.k_clean.numel() + (sb.k_donor.numel() if sb.k_donor is not None else 0)) * 4 / 1e9
    print(f"profile case ok: {wl.name}, {sb.B} sequences, step {args.step}, {wl.num_layers} layers, "
          f"{args.reps} reps, stores {gb:.2f} GB")
    return 0


if __name__ == "__main__":
    sys.exit(main())
