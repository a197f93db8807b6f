"""A random-initialised Qwen3-shaped decoder that drives spliced decode
attention end to end: Algorithm 1 (splice-intervention greedy decode) for a
whole sweep batch at once.

* Prefill (outside the decode hot path): every prompt of the batch and every
  stored donor of it (Table 1: BLANK, SAME_ALGO, DIFF_ALGO, DIFF_FAMILY token
  sequences of the prompt's length; ZERO is not stored) runs a full causal
  forward pass; its RoPE'd K and V fill the clean and donor stores the
  library reads, and the clean prompt's last logits give y_0.
* Decode: each step t = 1 .. T-1 runs one forward pass of every sequence's
  previous token y_{t-1} at position T_p + t - 1; at every layer one
  ``spliced_decode_step`` call appends the token's K/V to the generated-span
  store and lets the query attend over its prompt span -- clean, donor or
  ZERO by the splice rule l >= L and t >= W -- and its t generated entries;
  the last layer's output gives y_t = argmax.
  The replacement at t = W is not a copy: every sequence reads its source by
  reference, which is the same computation because the rule is monotone in t.

Real weights are out of scope: the weights are seeded random normals, so the
tokens mean nothing; what the run exercises is the propagation of the
splice through real forward passes (generated-span K/V that depend on the
spliced attention of every earlier layer and step), which the synthetic
inputs of the attention benchmark abstract away.  The projections, norms,
RoPE and MLP are plain torch (cuBLAS GEMMs); every decode attention is the
library's.
"""
from __future__ import annotations

import argparse
import math
import sys
import time
from dataclasses import dataclass
from typing import List, Optional, Sequence

import torch

from . import splice as S
from .synth import workloads as W


@dataclass(frozen=True)
class DecoderDims:
    num_layers: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    d_model: int
    ffn: int
    vocab: int
    rope_theta: float = 1.0e6
    rms_eps: float = 1.0e-6
    eos: Optional[int] = None


def qwen3_8b_dims() -> DecoderDims:
    """Qwen3-8B's published shape (36 layers, 32 / 8 heads of 128, d_model
    4096, MLP 12288, vocabulary 151936)."""
    return DecoderDims(36, 32, 8, 128, 4096, 12288, 151936)


def tiny_dims() -> DecoderDims:
    return DecoderDims(4, 8, 2, 64, 256, 512, 512)


def _rms_norm(x: torch.Tensor, w: torch.Tensor, eps: float) -> torch.Tensor:
    xf = x.float()
    return xf * torch.rsqrt(xf.pow(2).mean(-1, keepdim=True) + eps) * w.float()


class RandomDecoder:
    """Pre-norm decoder layers: RMSNorm -> q, k, v projections (GQA), per-head
    RMSNorm of q and k, RoPE -> attention -> output projection -> residual;
    RMSNorm -> SwiGLU MLP -> residual.  Final RMSNorm and LM head.  bf16
    weights, fp32 residual stream."""

    def __init__(self, dims: DecoderDims, seed: int = 0, device: str = "cuda", std: float = 0.02):
        self.dims = dims
        self.device = torch.device(device)
        g = torch.Generator(device=self.device)
        g.manual_seed(seed)
        bf = dict(dtype=torch.bfloat16, device=self.device)

        def rnd(*shape, scale=std):
            return (torch.randn(*shape, generator=g, dtype=torch.float32, device=self.device) * scale).to(torch.bfloat16)

        D, Hq, Hkv, d, F = dims.d_model, dims.num_q_heads, dims.num_kv_heads, dims.head_dim, dims.ffn
        self.embed = rnd(dims.vocab, D, scale=1.0)
        self.layers = []
        for _ in range(dims.num_layers):
            self.layers.append(dict(
                in_norm=torch.ones(D, **bf), wq=rnd(Hq * d, D), wk=rnd(Hkv * d, D), wv=rnd(Hkv * d, D),
                q_norm=torch.ones(d, **bf), k_norm=torch.ones(d, **bf), wo=rnd(D, Hq * d),
                post_norm=torch.ones(D, **bf), w_gate=rnd(F, D), w_up=rnd(F, D), w_down=rnd(D, F)))
        self.final_norm = torch.ones(D, **bf)
        self.lm_head = rnd(dims.vocab, D)
        half = d // 2
        self.inv_freq = 1.0 / (dims.rope_theta ** (torch.arange(half, device=self.device, dtype=torch.float32) / half))
        self.sm_scale = 1.0 / math.sqrt(d)

    # -- pieces -----------------------------------------------------------
    def rope(self, x: torch.Tensor, pos: torch.Tensor) -> torch.Tensor:
        """x [..., n, H, d] (fp32), pos [..., n] -> rotate-half RoPE."""
        ang = pos.float()[..., None] * self.inv_freq          # [..., n, d/2]
        cos, sin = ang.cos()[..., None, :], ang.sin()[..., None, :]
        h = x.shape[-1] // 2
        x1, x2 = x[..., :h], x[..., h:]
        return torch.cat([x1 * cos - x2 * sin, x2 * cos + x1 * sin], dim=-1)

    def qkv(self, l: int, h: torch.Tensor, pos: torch.Tensor):
        """h [..., n, D] fp32, pos [..., n] -> q [..., n, Hq, d], k, v [..., n, Hkv, d] (bf16)."""
        dims, w = self.dims, self.layers[l]
        x = _rms_norm(h, w["in_norm"], dims.rms_eps).to(torch.bfloat16)
        q = (x @ w["wq"].t()).unflatten(-1, (dims.num_q_heads, dims.head_dim))
        k = (x @ w["wk"].t()).unflatten(-1, (dims.num_kv_heads, dims.head_dim))
        v = (x @ w["wv"].t()).unflatten(-1, (dims.num_kv_heads, dims.head_dim))
        q = self.rope(_rms_norm(q, w["q_norm"], dims.rms_eps), pos)
        k = self.rope(_rms_norm(k, w["k_norm"], dims.rms_eps), pos)
        return q.to(torch.bfloat16), k.to(torch.bfloat16), v

    def block_out(self, l: int, h: torch.Tensor, attn: torch.Tensor) -> torch.Tensor:
        """Residual stream after layer l given its attention output attn [..., Hq, d]."""
        dims, w = self.dims, self.layers[l]
        h = h + (attn.to(torch.bfloat16).flatten(-2) @ w["wo"].t()).float()
        x = _rms_norm(h, w["post_norm"], dims.rms_eps).to(torch.bfloat16)
        gate = x @ w["w_gate"].t()
        up = x @ w["w_up"].t()
        return h + ((torch.nn.functional.silu(gate.float()) * up.float()).to(torch.bfloat16) @ w["w_down"].t()).float()

    def logits(self, h: torch.Tensor) -> torch.Tensor:
        x = _rms_norm(h, self.final_norm, self.dims.rms_eps).to(torch.bfloat16)
        return (x @ self.lm_head.t()).float()

    # -- prefill ----------------------------------------------------------
    @torch.no_grad()
    def prefill(self, tokens: torch.Tensor, k_out: torch.Tensor, v_out: torch.Tensor) -> torch.Tensor:
        """Causal forward of one token sequence [T_p] at positions 0..T_p-1.
        Writes every layer's RoPE'd K and V into k_out, v_out [N][Hkv][T_p][d]
        and returns the last position's logits [vocab]."""
        dims = self.dims
        G = dims.num_q_heads // dims.num_kv_heads
        pos = torch.arange(tokens.shape[0], device=self.device)
        h = self.embed[tokens].float()
        for l in range(dims.num_layers):
            q, k, v = self.qkv(l, h, pos)                   # [T_p, H, d]
            k_out[l].copy_(k.transpose(0, 1))
            v_out[l].copy_(v.transpose(0, 1))
            qh = q.transpose(0, 1)[None]                    # [1, Hq, T_p, d]
            kh = k.transpose(0, 1).repeat_interleave(G, dim=0)[None]
            vh = v.transpose(0, 1).repeat_interleave(G, dim=0)[None]
            a = torch.nn.functional.scaled_dot_product_attention(qh, kh, vh, is_causal=True, scale=self.sm_scale)
            h = self.block_out(l, h, a[0].transpose(0, 1).float())
        return self.logits(h[-1])


def donor_tokens(prompt: torch.Tensor, kind: int, gen: torch.Generator, vocab: int, scaffold_head: int,
                 scaffold_tail: int, filler: int) -> Optional[torch.Tensor]:
    """Token sequence of a donor of the prompt (Table 1), same length: the
    scaffold (first / last positions) is kept; BLANK fills the content with
    one filler token; SAME_ALGO / DIFF_ALGO replace a fixed fraction of the
    content positions (0.1 / 0.5, the ladder's) with other tokens;
    DIFF_FAMILY draws fresh content.  ZERO has no tokens (all-zero K, V)."""
    if kind == W.ZERO:
        return None
    Tp = prompt.shape[0]
    out = prompt.clone()
    lo, hi = min(scaffold_head, Tp), max(min(scaffold_head, Tp), Tp - scaffold_tail)
    content = torch.arange(lo, hi, device=prompt.device)
    if content.numel() == 0:
        return out
    fresh = torch.randint(0, vocab, (content.numel(),), generator=gen, device=prompt.device)
    if kind == W.BLANK:
        out[content] = filler
    elif kind == W.DIFF_FAMILY:
        out[content] = fresh
    else:
        frac = W.PERTURB_THRESHOLD_24[kind] / float(1 << 24)
        pick = torch.rand(content.numel(), generator=gen, device=prompt.device) < frac
        out[content[pick]] = fresh[pick]
    return out


class SpliceDecode:
    """Algorithm 1 for a batch of sweep cells (prompt, donor slot, L, W) with
    a random decoder.  Holds the prompt and donor stores (from prefill), the
    generated-span store, the descriptor and the workspace."""

    def __init__(self, model: RandomDecoder, prompts: torch.Tensor, slot_kinds: Sequence[int],
                 seqs: Sequence[W.Seq], max_steps: int, scaffold_head: int = 0, scaffold_tail: int = 0,
                 filler: int = 0, seed: int = 0):
        """prompts [P][T_p] token ids; seqs index prompts 0..P-1 and slots of slot_kinds."""
        dims, dev = model.dims, model.device
        self.model, self.seqs, self.T = model, list(seqs), max_steps
        P, Tp = prompts.shape
        self.P, self.Tp, self.B = P, Tp, len(self.seqs)
        self.slot_kinds = tuple(slot_kinds)
        self.stored = [k for k, kd in enumerate(self.slot_kinds) if kd != W.ZERO]
        N, Hkv, d = dims.num_layers, dims.num_kv_heads, dims.head_dim
        bf = dict(dtype=torch.bfloat16, device=dev)
        self.k_clean = torch.empty((P, N, Hkv, Tp, d), **bf)
        self.v_clean = torch.empty_like(self.k_clean)
        Dst = len(self.stored)
        self.k_donor = torch.empty((P, Dst, N, Hkv, Tp, d), **bf) if Dst else None
        self.v_donor = torch.empty_like(self.k_donor) if Dst else None
        gen = torch.Generator(device=dev)
        gen.manual_seed(seed + 1)
        self.y0 = torch.empty(P, dtype=torch.long, device=dev)
        self.donor_prompts = {}
        for p in range(P):
            self.y0[p] = model.prefill(prompts[p], self.k_clean[p], self.v_clean[p]).argmax()
            for i, k in enumerate(self.stored):
                toks = donor_tokens(prompts[p], self.slot_kinds[k], gen, dims.vocab, scaffold_head, scaffold_tail,
                                    filler)
                self.donor_prompts[(p, k)] = toks
                model.prefill(toks, self.k_donor[p, i], self.v_donor[p, i])
        self.k_suffix = torch.zeros((self.B, N, Hkv, max_steps, d), **bf)
        self.v_suffix = torch.zeros_like(self.k_suffix)
        shape = dict(num_layers=N, num_q_heads=dims.num_q_heads, num_kv_heads=Hkv, head_dim=d,
                     sliding_window=0, global_every=0, sm_scale=model.sm_scale)
        self.desc = S.splice_desc_create(shape, P, Tp, self.slot_kinds,
                                         [(q.prompt, q.slot, q.L, q.W) for q in self.seqs], max_steps)
        self.ws = torch.empty(S.splice_workspace_bytes(self.desc), dtype=torch.uint8, device=dev)
        self.out = torch.empty((self.B, dims.num_q_heads, d), dtype=torch.float32, device=dev)
        self.first_token = self.y0[torch.tensor([q.prompt for q in self.seqs], device=dev)]

    @torch.no_grad()
    def step(self, t: int, tokens: torch.Tensor) -> torch.Tensor:
        """Forward pass of step t (1 <= t < T): tokens [B] are y_{t-1}; returns
        the logits [B][vocab] whose argmax is y_t."""
        model, dims = self.model, self.model.dims
        pos = torch.full((self.B,), self.Tp + t - 1, device=model.device)
        h = model.embed[tokens].float()
        for l in range(dims.num_layers):
            q, k, v = model.qkv(l, h, pos)
            S.spliced_decode_step(self.desc, l, t, q.contiguous(), k.contiguous(), v.contiguous(), self.k_clean,
                                  self.v_clean, self.k_donor, self.v_donor, self.k_suffix, self.v_suffix, self.out,
                                  self.ws)
            h = model.block_out(l, h, self.out)
        return model.logits(h)

    @torch.no_grad()
    def decode(self, steps: Optional[int] = None) -> torch.Tensor:
        """Greedy splice-intervention decode; returns tokens [B][steps]
        (y_0 .. y_{steps-1}); after a sequence's eos its later tokens are eos."""
        steps = self.T if steps is None else steps
        toks = [self.first_token]
        done = torch.zeros(self.B, dtype=torch.bool, device=self.model.device)
        eos = self.model.dims.eos
        for t in range(1, steps):
            y = self.step(t, toks[-1]).argmax(-1)
            if eos is not None:
                done |= toks[-1] == eos
                y = torch.where(done, torch.full_like(y, eos), y)
            toks.append(y)
        S.splice_check_device_error(self.desc)
        return torch.stack(toks, dim=1)

    def close(self):
        self.desc.close()


def ladder_batch_cells(wl: W.Workload, batch: int = 0) -> List[W.Seq]:
    lo, hi = wl.batch_range(batch)
    return wl.sequences()[lo:hi]


def main(argv=None):
    """Times Algorithm 1 for a Qwen3-8B-shaped random decoder on batch 0 of the
    ladder sweep (its cells, prompt length and donor kinds)."""
    ap = argparse.ArgumentParser(description=main.__doc__)
    ap.add_argument("--steps", type=int, default=16, help="decode steps timed (after the warm-up)")
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--prompt-len", type=int, default=None)
    ap.add_argument("--workload", default="qwen3-8b-ladder")
    args = ap.parse_args(argv)
    from . import build as B
    B.build()
    import json
    wl = W.get(args.workload)
    dims = qwen3_8b_dims()
    seqs = ladder_batch_cells(wl, 0)
    p0 = min(q.prompt for q in seqs)
    seqs = [W.Seq(q.prompt - p0, q.slot, q.L, q.W) for q in seqs]
    P = max(q.prompt for q in seqs) + 1
    Tp = args.prompt_len or wl.prompt_len
    T = args.warmup + args.steps + 1
    model = RandomDecoder(dims, seed=0)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(7)
    prompts = torch.randint(0, dims.vocab, (P, Tp), generator=gen, device="cuda")
    t0 = time.time()
    run = SpliceDecode(model, prompts, wl.slot_kinds, seqs, T, wl.scaffold_head, wl.scaffold_tail, filler=64)
    torch.cuda.synchronize()
    prefill_s = time.time() - t0
    toks = run.first_token
    for t in range(1, args.warmup + 1):
        toks = run.step(t, toks).argmax(-1)
    torch.cuda.synchronize()
    timed = list(range(args.warmup + 1, args.warmup + 1 + args.steps))
    inputs = []
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record()
    for t in timed:
        inputs.append(toks)
        toks = run.step(t, toks).argmax(-1)
    ev1.record()
    torch.cuda.synchronize()
    ms = ev0.elapsed_time(ev1)
    # the attention's share: the same steps again with the library's
    # per-launch timing on (its launches then run one after another)
    S.splice_profile_enable(run.desc, True)
    S.splice_profile_read(run.desc)
    for t, tin in zip(timed, inputs):
        run.step(t, tin)
    torch.cuda.synchronize()
    prof = S.splice_profile_read(run.desc)
    S.splice_profile_enable(run.desc, False)
    S.splice_check_device_error(run.desc)
    attn_ms = sum(v[1] for v in prof.values())
    print(json.dumps({
        "what": "Algorithm 1 greedy decode, random-init Qwen3-8B-shaped decoder, ladder batch 0",
        "sequences": run.B, "prompts": P, "prompt_len": Tp, "donor_slots": len(wl.slot_kinds),
        "steps_timed": args.steps, "ms_per_step": round(ms / args.steps, 3),
        "tokens_per_s": round(run.B * args.steps / (ms / 1e3), 1),
        "library_ms_per_step_serialised": round(attn_ms / args.steps, 3),
        "library_kernels": {k: round(v[1] / args.steps, 3) for k, v in prof.items()},
        "prefill_s": round(prefill_s, 2)}))
    run.close()
    return 0


if __name__ == "__main__":
    sys.exit(main())
