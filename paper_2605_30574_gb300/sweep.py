"""One decode batch of an (L, W, donor) sweep, resident on the GPU.

Allocates the stores the C ABI reads (clean prompt spans and stored donor
spans of the batch's prompts, every sequence's generated-span store), fills
them with the seeded device generator, builds the splice descriptor, and
drives ``suffix_kv_append`` + ``spliced_decode_attn`` for a (layer, step).
Torch only owns memory and streams here.
"""
from __future__ import annotations

import torch

from . import splice as S
from .synth import device as SD
from .synth import workloads as W


def model_shape(wl: W.Workload) -> dict:
    return dict(num_layers=wl.num_layers, num_q_heads=wl.num_q_heads, num_kv_heads=wl.num_kv_heads,
                head_dim=wl.head_dim, sliding_window=wl.sliding_window, global_every=wl.global_every,
                sm_scale=wl.sm_scale)


class SweepBatch:
    def __init__(self, wl: W.Workload, batch: int = 0, device: str = "cuda", fill: bool = True,
                 seqs=None):
        """``seqs``: explicit list of Seq (global prompt ids, sequence ids 0..len-1)
        instead of batch ``batch`` of the workload's enumerated sweep."""
        self.wl = wl
        if seqs is None:
            lo, hi = wl.batch_range(batch)
            self.seqs = wl.sequences()[lo:hi]
            c = wl.cells_per_prompt()
            self.p0 = lo // c
            self.Pl = (hi - 1) // c + 1 - self.p0
        else:
            lo, hi = 0, len(seqs)
            self.seqs = list(seqs)
            self.p0 = min(q.prompt for q in self.seqs)
            self.Pl = max(q.prompt for q in self.seqs) + 1 - self.p0
        self.s0, self.B = lo, hi - lo
        self.Dst = sum(1 for k in wl.slot_kinds if k != W.ZERO)
        N, Hq, Hkv, d, Tp, T = (wl.num_layers, wl.num_q_heads, wl.num_kv_heads, wl.head_dim,
                                wl.prompt_len, wl.max_steps)
        bf = dict(dtype=torch.bfloat16, device=device)
        self.k_clean = torch.empty((self.Pl, N, Hkv, Tp, d), **bf)
        self.v_clean = torch.empty_like(self.k_clean)
        if self.Dst:
            self.k_donor = torch.empty((self.Pl, self.Dst, N, Hkv, Tp, d), **bf)
            self.v_donor = torch.empty_like(self.k_donor)
        else:
            self.k_donor = self.v_donor = None
        self.k_suffix = torch.empty((self.B, N, Hkv, T, d), **bf)
        self.v_suffix = torch.empty_like(self.k_suffix)
        self.q = torch.empty((self.B, Hq, d), **bf)
        self.k_new = torch.empty((self.B, Hkv, d), **bf)
        self.v_new = torch.empty_like(self.k_new)
        self.out = torch.empty((self.B, Hq, d), dtype=torch.float32, device=device)
        self.desc = S.splice_desc_create(model_shape(wl), self.Pl, Tp, wl.slot_kinds,
                                         [(q.prompt - self.p0, q.slot, q.L, q.W) for q in self.seqs], T)
        self.ws = torch.empty(S.splice_workspace_bytes(self.desc), dtype=torch.uint8, device=device)
        if fill:
            self.fill()

    def fill(self):
        SD.fill_clean(self.wl, self.p0, self.k_clean, self.v_clean)
        if self.Dst:
            SD.fill_donor(self.wl, self.p0, self.k_donor, self.v_donor)
        SD.fill_suffix(self.wl, self.s0, self.k_suffix, self.v_suffix)

    def gen_inputs(self, layer: int, step: int, q=None, k_new=None, v_new=None):
        """Generate the queries and this step's generated K/V of (layer, step)."""
        q = self.q if q is None else q
        k_new = self.k_new if k_new is None else k_new
        v_new = self.v_new if v_new is None else v_new
        SD.fill_q(self.wl, self.s0, layer, step, q)
        if step >= 1:
            SD.fill_new_kv(self.wl, self.s0, layer, step, k_new, v_new)

    def append(self, layer: int, step: int, k_new=None, v_new=None, stream=None):
        S.suffix_kv_append(self.desc, layer, step, self.k_new if k_new is None else k_new,
                           self.v_new if v_new is None else v_new, self.k_suffix, self.v_suffix, stream)

    def attn(self, layer: int, step: int, q=None, out=None, stream=None):
        S.spliced_decode_attn(self.desc, layer, step, self.q if q is None else q, self.k_clean, self.v_clean,
                              self.k_donor, self.v_donor, self.k_suffix, self.v_suffix,
                              self.out if out is None else out, self.ws, stream=stream)

    def step(self, layer: int, step: int, q=None, k_new=None, v_new=None, out=None, stream=None):
        """The fused call: append this step's K/V and attend (step >= 1)."""
        S.spliced_decode_step(self.desc, layer, step, self.q if q is None else q,
                              self.k_new if k_new is None else k_new, self.v_new if v_new is None else v_new,
                              self.k_clean, self.v_clean, self.k_donor, self.v_donor, self.k_suffix, self.v_suffix,
                              self.out if out is None else out, self.ws, stream=stream)

    def run(self, layer: int, step: int):
        """Generate inputs, append (step >= 1) and attend; returns self.out."""
        self.gen_inputs(layer, step)
        if step >= 1:
            self.append(layer, step)
        self.attn(layer, step)
        return self.out

    def close(self):
        self.desc.close()
