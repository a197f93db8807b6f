"""Sweep reporting: the L x W phase diagram of one intervention and its
recovery frontier (§3 "Sweep and reporting"; Appendix "Clean Baselines").

For one condition (model, task, donor kind) the sweep gives a pass rate
pass(L, W) for every cell of the grid.  The phase diagram is that rate laid
out over L x W; the recovery frontier at a threshold alpha in (0, 1] is, for
every cutoff L, the least onset W whose pass rate reaches alpha times the
unintervened pass rate p_clean:

    W*(L; alpha) = min { W : pass(L, W) >= alpha * p_clean }

(None where no W of the grid reaches it).

Pass rates need a task and a scorer.  The paper scores benchmark items with
real models, which are out of reach here; ``decode_pass_rates`` scores the
random-initialised decoder of ``model.py`` instead: a cell passes when its
greedy continuation is token for token the unintervened continuation of the
same prompt (exact match), or, with ``match="token"``, by the fraction of its
tokens that agree.  The tokens of a random decoder mean nothing, so such a
diagram says how far a splice moves the decode, not whether a task is solved.

``python -m paper_2605_30574_gb300.report`` runs that sweep on the GPU
(every decode attention through the library) and prints the diagrams and
frontiers; the functions above it are plain host code.
"""
from __future__ import annotations

import argparse
import json
import math
import sys
from typing import Dict, List, Mapping, Optional, Sequence, Tuple

import numpy as np

from .synth import workloads as W


def phase_grid(rates: Mapping[Tuple[int, int], float], Ls: Sequence[int], Ws: Sequence[int]) -> np.ndarray:
    """pass(L, W) on the grid: [len(Ls)][len(Ws)], NaN where a cell has no rate."""
    g = np.full((len(Ls), len(Ws)), np.nan)
    for i, L in enumerate(Ls):
        for j, Wv in enumerate(Ws):
            if (L, Wv) in rates:
                g[i, j] = rates[(L, Wv)]
    return g


def recovery_frontier(grid: np.ndarray, Ws: Sequence[int], p_clean: float, alpha: float) -> List[Optional[int]]:
    """W*(L; alpha) for every row of ``grid`` (one row per L, columns in the
    order of ``Ws``, which need not be sorted): the least W whose rate is at
    least alpha * p_clean; None where none is.  Cells without a rate (NaN)
    never qualify."""
    if not 0.0 < alpha <= 1.0:
        raise ValueError("alpha must lie in (0, 1]")
    grid = np.asarray(grid, dtype=np.float64)
    if grid.ndim != 2 or grid.shape[1] != len(Ws):
        raise ValueError("grid must be [len(Ls)][len(Ws)]")
    need = alpha * p_clean
    out: List[Optional[int]] = []
    for row in grid:
        ok = [Wv for Wv, r in zip(Ws, row) if not math.isnan(r) and r >= need]
        out.append(min(ok) if ok else None)
    return out


def render_grid(grid: np.ndarray, Ls: Sequence[int], Ws: Sequence[int], title: str = "") -> str:
    """Text heatmap: rows L, columns W, pass rates in percent ('.' = no rate)."""
    w = max(4, max(len(str(x)) for x in Ws) + 1)
    lines = [title] if title else []
    lines.append("L \\ W".rjust(6) + "".join(str(x).rjust(w) for x in Ws))
    for L, row in zip(Ls, grid):
        cells = "".join(("." if math.isnan(r) else f"{100.0 * r:.0f}").rjust(w) for r in row)
        lines.append(str(L).rjust(6) + cells)
    return "\n".join(lines)


def render_frontiers(frontiers: Mapping[str, Sequence[Optional[int]]], Ls: Sequence[int], title: str = "") -> str:
    """Table of W*(L) per condition ('-' where no W of the grid recovers)."""
    names = list(frontiers)
    w = max(8, max((len(n) for n in names), default=0) + 2)
    lines = [title] if title else []
    lines.append("L".rjust(6) + "".join(n.rjust(w) for n in names))
    for i, L in enumerate(Ls):
        lines.append(str(L).rjust(6) + "".join(
            ("-" if frontiers[n][i] is None else str(frontiers[n][i])).rjust(w) for n in names))
    return "\n".join(lines)


def decode_pass_rates(tokens: np.ndarray, seqs: Sequence[W.Seq], reference: Mapping[int, int],
                      match: str = "exact") -> Dict[Tuple[int, int, int], float]:
    """Pass rate per (slot, L, W) over prompts.

    tokens [B][T] are the greedy continuations of the cells ``seqs`` (row b
    is cell b); ``reference`` maps a prompt to the row of its unintervened
    continuation.  ``match="exact"`` scores a cell 1 when its row equals the
    reference row, else 0; ``match="token"`` scores the fraction of equal
    tokens.  The rate of (slot, L, W) is the mean score of its cells; the
    reference rows themselves are not cells of the grid."""
    tokens = np.asarray(tokens)
    if match not in ("exact", "token"):
        raise ValueError("match must be 'exact' or 'token'")
    ref_rows = set(reference.values())
    acc: Dict[Tuple[int, int, int], List[float]] = {}
    for b, q in enumerate(seqs):
        if b in ref_rows:
            continue
        ref = tokens[reference[q.prompt]]
        eq = tokens[b] == ref
        score = float(eq.all()) if match == "exact" else float(eq.mean())
        acc.setdefault((q.slot, q.L, q.W), []).append(score)
    return {k: float(np.mean(v)) for k, v in acc.items()}


def sweep_cells(num_prompts: int, num_slots: int, Ls: Sequence[int], Ws: Sequence[int],
                num_layers: int) -> Tuple[List[W.Seq], Dict[int, int]]:
    """Cells of a decode sweep: for every prompt one unintervened cell
    (L = num_layers patches no layer) followed by every (slot, L, W) of the
    grid; returns the cells and each prompt's unintervened row."""
    seqs: List[W.Seq] = []
    reference: Dict[int, int] = {}
    for p in range(num_prompts):
        reference[p] = len(seqs)
        seqs.append(W.Seq(p, 0, num_layers, 0))
        for k in range(num_slots):
            for L in Ls:
                for Wv in Ws:
                    seqs.append(W.Seq(p, k, L, Wv))
    return seqs, reference


def run_decode_sweep(dims, slot_kinds: Sequence[int], Ls: Sequence[int], Ws: Sequence[int], num_prompts: int,
                     prompt_len: int, steps: int, seed: int = 0, scaffold_head: int = 24, scaffold_tail: int = 12,
                     filler: int = 64):
    """Greedy splice-intervention decode of every cell of the grid with a
    random decoder of shape ``dims`` (GPU).  Returns (tokens [B][steps] on the
    host, cells, reference rows)."""
    import torch

    from .model import RandomDecoder, SpliceDecode
    seqs, reference = sweep_cells(num_prompts, len(slot_kinds), Ls, Ws, dims.num_layers)
    model = RandomDecoder(dims, seed=seed)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(seed + 7)
    prompts = torch.randint(0, dims.vocab, (num_prompts, prompt_len), generator=gen, device="cuda")
    run = SpliceDecode(model, prompts, slot_kinds, seqs, steps, scaffold_head, scaffold_tail, filler, seed=seed)
    try:
        toks = run.decode(steps).cpu().numpy()
    finally:
        run.close()
    return toks, seqs, reference


def report(tokens: np.ndarray, seqs: Sequence[W.Seq], reference: Mapping[int, int], slot_kinds: Sequence[int],
           Ls: Sequence[int], Ws: Sequence[int], alphas: Sequence[float], match: str = "exact") -> dict:
    """Phase diagrams and frontiers of a decode sweep, one condition per donor
    slot.  The unintervened decode is its own reference, so p_clean = 1 under
    both scores."""
    rates = decode_pass_rates(tokens, seqs, reference, match)
    p_clean = 1.0
    out = {"match": match, "p_clean": p_clean, "Ls": list(Ls), "Ws": list(Ws), "conditions": {}}
    for k, kind in enumerate(slot_kinds):
        g = phase_grid({(L, Wv): r for (s, L, Wv), r in rates.items() if s == k}, Ls, Ws)
        out["conditions"][W.KIND_NAMES[kind]] = {
            "grid": [[None if math.isnan(x) else x for x in row] for row in g],
            "frontier": {str(a): recovery_frontier(g, Ws, p_clean, a) for a in alphas},
        }
    return out


def main(argv=None) -> int:
    """Decode sweep with a random-initialised decoder; prints each donor
    kind's phase diagram and the recovery frontiers."""
    ap = argparse.ArgumentParser(description=main.__doc__)
    ap.add_argument("--dims", choices=("tiny", "qwen3-8b"), default="tiny")
    ap.add_argument("--prompts", type=int, default=4)
    ap.add_argument("--prompt-len", type=int, default=128)
    ap.add_argument("--steps", type=int, default=32, help="tokens generated per cell (y_0 .. y_{steps-1})")
    ap.add_argument("--L-step", type=int, default=None, help="L grid stride (default: 3 for qwen3-8b, 1 for tiny)")
    ap.add_argument("--W", type=int, nargs="+", default=None, help="W grid (default 0, 2, 4, ... below steps)")
    ap.add_argument("--alpha", type=float, nargs="+", default=[0.4, 0.67, 0.75])
    ap.add_argument("--kinds", nargs="+", default=["BLANK", "ZERO", "SAME_ALGO", "DIFF_ALGO", "DIFF_FAMILY"])
    ap.add_argument("--match", choices=("exact", "token"), default="exact")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--json", default=None, help="also write the report here")
    args = ap.parse_args(argv)
    from . import build as B
    from .model import qwen3_8b_dims, tiny_dims
    B.build()
    dims = qwen3_8b_dims() if args.dims == "qwen3-8b" else tiny_dims()
    step = args.L_step or (3 if args.dims == "qwen3-8b" else 1)
    Ls = sorted(set(list(range(0, dims.num_layers, step)) + [dims.num_layers]))
    Ws = args.W or list(range(0, args.steps, max(1, args.steps // 8)))
    names = {v: k for k, v in W.KIND_NAMES.items()}
    kinds = [names[k] for k in args.kinds]
    head, tail = (24, 12) if args.dims == "qwen3-8b" else (4, 2)
    toks, seqs, ref = run_decode_sweep(dims, kinds, Ls, Ws, args.prompts, args.prompt_len, args.steps,
                                       seed=args.seed, scaffold_head=head, scaffold_tail=tail)
    rep = report(toks, seqs, ref, kinds, Ls, Ws, args.alpha, args.match)
    rep.update({"dims": args.dims, "prompts": args.prompts, "prompt_len": args.prompt_len, "steps": args.steps,
                "cells": len(seqs)})
    for name, c in rep["conditions"].items():
        g = np.array([[np.nan if x is None else x for x in row] for row in c["grid"]])
        print(render_grid(g, Ls, Ws, f"{name}: pass(L, W) % ({args.match} match vs the unintervened decode)"))
        print()
    for a in args.alpha:
        print(render_frontiers({n: c["frontier"][str(a)] for n, c in rep["conditions"].items()}, Ls,
                               f"recovery frontier W*(L; alpha={a})"))
        print()
    if args.json:
        with open(args.json, "w") as f:
            json.dump(rep, f)
    return 0


if __name__ == "__main__":
    sys.exit(main())
