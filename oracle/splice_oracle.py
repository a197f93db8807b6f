"""CPU fp64 oracle for spliced decode attention (arxiv 2605.30574, §3).

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import or call
this module: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it.  It shares
no code with the CUDA path; the seeded input generator
(``paper_2605_30574_gb300.synth``) is the only module both read.

What it computes, step by step, the slow and obvious way:

1. ``splice_source`` -- which prompt-span K/V a sequence reads at layer l and
   decode step t (§3 "Splice intervention"; Algorithm 1).  The patched layer
   set is {l : l >= L}; the replacement happens at step t = W and persists to
   the end of decoding, so layer l at step t reads the donor iff l >= L and
   t >= W.  Steps are Algorithm 1's loop variable t = 1..T; W = 0 means the
   span is replaced before the first step (reading A1: W = 0 and W = 1 give
   the same run).  A ZERO donor (Table 1) is the all-zero K, V.
2. ``spliced_prompt_kv`` -- an explicit *copy* of that span (clean, donor or
   zeros) into a fresh buffer, as the in-place replacement of §3 would leave
   the cache.
3. ``decode_attn`` -- appends the sequence's own generated-span entries
   0..t-1 (§3: the decoding step attends over the prompt span concatenated
   with the generated span; generated entries are never modified; the
   current token's own K/V is appended before attention, Algorithm 1's
   forward pass) and runs naive softmax attention in fp64 from the exact bf16
   values: kv head of q head h is floor(h / G); on sliding-window layers a
   key at absolute position j is visible iff (T_p + t - 1) - j < window.
4. ``partial`` / ``merge_partials`` -- the log-sum-exp combination of
   attention over disjoint key sets (the merge step of the path).  It is the
   standard identity softmax over a union = weighted combination of
   per-part softmaxes; pinned against single-pass softmax in the tests.

5. ``delta_positions`` / ``delta_encode`` / ``delta_decode`` -- the
   delta encoding of a stored donor span against the clean span of the same
   prompt, layer and kv head: the positions whose K row or V row differs bit
   for bit, and the donor rows at those positions in increasing position
   order.  Table 1's donors are positionally aligned with the clean prompt
   (§3: scaffolds are trimmed to the same length), so a donor shares every
   position whose rows are equal; the encoding is lossless by definition
   (``delta_decode`` rebuilds the donor span exactly), and attention over
   the donor span is the merge of attention over the clean span without
   those positions and over the encoded rows (step 4).

Parity is pinned (tests/test_oracle_pins.py) by hand-derived cases
(tests/golden/), a literal in-place simulation of Algorithm 1, the ZERO
closed form, torch's CPU scaled_dot_product_attention on materialised
caches, and LSE-merge identities.  No pin links it to the paper's accuracy
numbers (they need model weights and datasets): those are out of scope.
"""
from __future__ import annotations

import numpy as np

# Source codes, the same meaning as the C ABI's debug source map.
SRC_CLEAN = 0
SRC_ZERO = 1
SRC_DONOR0 = 2      # donor slot k -> 2 + k

KIND_ZERO = 0       # Table 1 ZERO; every other kind is a stored donor cache


def splice_source(L: int, W: int, slot: int, slot_kind: int, l: int, t: int) -> int:
    """Prompt-span source of layer l at decode step t for cell (slot, L, W).

    §3: layers in P = {l >= L} are patched; steps t < W use the clean cache
    and the replacement made at t = W persists (Algorithm 1).
    """
    if l >= L and t >= W:
        return SRC_ZERO if slot_kind == KIND_ZERO else SRC_DONOR0 + slot
    return SRC_CLEAN


def layer_is_global(l: int, window: int, global_every: int) -> bool:
    if window <= 0:
        return True
    if global_every <= 0:
        return False
    return (l + 1) % global_every == 0


def visible_range(prompt_len: int, t: int, l: int, window: int, global_every: int):
    """[lo, hi) of absolute key positions visible to the step-t query.

    The query sits at absolute position prompt_len + t - 1 and the cache holds
    prompt_len + t entries.  Sliding-window layers keep keys with
    (query position - j) < window (the window includes the query itself).
    """
    hi = prompt_len + t
    lo = 0
    if not layer_is_global(l, window, global_every):
        lo = max(0, prompt_len + t - 1 - window + 1)
    return lo, hi


def bf16_to_f64(u) -> np.ndarray:
    """Exact value of bf16 bit patterns (uint16) as fp64."""
    u = np.asarray(u, dtype=np.uint16)
    return (u.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def spliced_prompt_kv(src: int, clean_k, clean_v, donor_k=None, donor_v=None):
    """Copy the prompt span the sequence reads into fresh fp64 arrays [Hkv][T_p][d]."""
    if src == SRC_CLEAN:
        return bf16_to_f64(clean_k).copy(), bf16_to_f64(clean_v).copy()
    if src == SRC_ZERO:
        shape = np.asarray(clean_k).shape
        return np.zeros(shape, np.float64), np.zeros(shape, np.float64)
    return bf16_to_f64(donor_k).copy(), bf16_to_f64(donor_v).copy()


def attend(q: np.ndarray, K: np.ndarray, V: np.ndarray, lo: int, sm_scale: float) -> np.ndarray:
    """Softmax attention of every q head over cache entries [lo, n).

    q: [Hq][d] fp64; K, V: [Hkv][n][d] fp64.  Returns [Hq][d] fp64.  With no
    visible entry the output row is 0.
    """
    Hq, d = q.shape
    Hkv = K.shape[0]
    G = Hq // Hkv
    out = np.zeros((Hq, V.shape[2]), np.float64)
    for h in range(Hq):
        kv = h // G
        Kh = K[kv, lo:]
        if Kh.shape[0] == 0:
            continue
        z = sm_scale * (Kh @ q[h])
        w = np.exp(z - z.max())
        out[h] = (w @ V[kv, lo:]) / w.sum()
    return out


def decode_attn(wl, inputs, s: int, seq, l: int, t: int) -> np.ndarray:
    """Spliced decode attention of sequence ``seq`` (global index s) at layer l, step t.

    ``wl`` carries the shapes (a synth Workload or any object with the same
    fields); ``inputs`` provides bf16 tensors: ``q(s, t, l)`` [Hq][d],
    ``clean_kv(p, l)``, ``donor_kv(p, k, l)`` [Hkv][T_p][d] and
    ``suffix_kv(s, l, 0, t)`` [Hkv][t][d].  Returns out [Hq][d] in fp64.
    """
    kind = wl.slot_kinds[seq.slot]
    src = splice_source(seq.L, seq.W, seq.slot, kind, l, t)
    ck, cv = inputs.clean_kv(seq.prompt, l)
    dk = dv = None
    if src >= SRC_DONOR0:
        dk, dv = inputs.donor_kv(seq.prompt, seq.slot, l)
    Kp, Vp = spliced_prompt_kv(src, ck, cv, dk, dv)
    sk, sv = inputs.suffix_kv(s, l, 0, t)
    K = np.concatenate([Kp, bf16_to_f64(sk)], axis=1)
    V = np.concatenate([Vp, bf16_to_f64(sv)], axis=1)
    lo, hi = visible_range(wl.prompt_len, t, l, wl.sliding_window, wl.global_every)
    assert hi == K.shape[1]
    q = bf16_to_f64(inputs.q(s, t, l))
    return attend(q, K, V, lo, wl.sm_scale)


def partial(q_row: np.ndarray, K: np.ndarray, V: np.ndarray, sm_scale: float):
    """Unnormalised attention of one query row over one key set: (m, l, o).

    m = max logit, l = sum exp(z - m), o = sum exp(z - m) V.  An empty key set
    gives (-inf, 0, 0).
    """
    if K.shape[0] == 0:
        return -np.inf, 0.0, np.zeros(V.shape[1], np.float64)
    z = sm_scale * (K @ q_row)
    m = z.max()
    w = np.exp(z - m)
    return m, w.sum(), w @ V


def merge_partials(parts):
    """Log-sum-exp merge: out = sum e^(m_i - M) o_i / sum e^(m_i - M) l_i, M = max m_i."""
    live = [p for p in parts if p[1] > 0]
    if not live:
        return np.zeros_like(parts[0][2])
    M = max(p[0] for p in live)
    num = sum(np.exp(m - M) * o for m, _, o in live)
    den = sum(np.exp(m - M) * l for m, l, _ in live)
    return num / den


def delta_positions(clean_k, clean_v, donor_k, donor_v) -> np.ndarray:
    """Positions of one span [T_p][d] (bf16 bit patterns) where the donor
    differs from the clean span: bool [T_p], True where the K row or the V
    row is not equal bit for bit."""
    ck, cv = np.asarray(clean_k, np.uint16), np.asarray(clean_v, np.uint16)
    dk, dv = np.asarray(donor_k, np.uint16), np.asarray(donor_v, np.uint16)
    return (ck != dk).any(axis=1) | (cv != dv).any(axis=1)


def delta_encode(clean_k, clean_v, donor_k, donor_v):
    """(mask [T_p] bool, rows_k [n][d], rows_v [n][d]): the differing
    positions and the donor's rows there, in increasing position order."""
    mask = delta_positions(clean_k, clean_v, donor_k, donor_v)
    idx = np.nonzero(mask)[0]
    return mask, np.asarray(donor_k, np.uint16)[idx].copy(), np.asarray(donor_v, np.uint16)[idx].copy()


def delta_decode(clean_k, clean_v, mask, rows_k, rows_v):
    """The donor span rebuilt from the clean span and its delta encoding."""
    k = np.array(clean_k, np.uint16, copy=True)
    v = np.array(clean_v, np.uint16, copy=True)
    idx = np.nonzero(np.asarray(mask, bool))[0]
    k[idx] = rows_k
    v[idx] = rows_v
    return k, v


def pack_mask_words(mask, words: int) -> np.ndarray:
    """Bit j % 32 of word j // 32 set iff mask[j]; ``words`` uint32 words."""
    out = np.zeros(words, np.uint32)
    for j in np.nonzero(np.asarray(mask, bool))[0]:
        out[j // 32] |= np.uint32(1) << np.uint32(j % 32)
    return out
