"""Host (numpy) twin of the seeded synthetic-input generator.

Every input value of the spliced decode-attention workloads is a pure
function of its logical coordinates, so any element can be regenerated on
the host without materialising whole tensors.  The device twin
(``synth.cu``) implements the same definition bit for bit; tests compare the
two on sampled coordinates.  Nothing here is part of the method: the splice
rule and the attention arithmetic live in the CUDA path and, separately, in
the oracle.

Definition
----------
* Counter-based draws use splitmix64 (Steele, Lea & Flood, OOPSLA 2014; the
  64-bit finaliser with multipliers 0xBF58476D1CE4E5B9 / 0x94D049BB133111EB
  and increment 0x9E3779B97F4A7C15).  ``mix`` is the finaliser.
* A stream ``(seed, stream_id)`` is the splitmix64 sequence whose state is
  ``x0 = mix(seed * 256 + stream_id + GAMMA)``; element ``i`` of the stream
  is ``mix(x0 + (i + 1) * GAMMA)`` (all mod 2**64), i.e. output i of a
  splitmix64 generator seeded with x0.
* An approximately N(0, 1) value is drawn from the four 16-bit fields of
  one 64-bit output: ``c = sum(fields) - 131070`` (exact integer), then
  ``z = f32(c) * f32(1 / 37837.2272...)`` rounded to fp32 (the sum of four
  uniforms on {0..65535} has standard deviation sqrt(4 (65536^2 - 1) / 12)).
  A value with multiplier ``a`` (fp32) is ``bf16_rne(f32(z * a))``.
* Element index = the row-major linear index of the logical coordinates
  listed for each stream below.
"""
from __future__ import annotations

import numpy as np

from . import workloads as W

GAMMA = np.uint64(0x9E3779B97F4A7C15)
MIX1 = np.uint64(0xBF58476D1CE4E5B9)
MIX2 = np.uint64(0x94D049BB133111EB)
NORMAL_SCALE_BITS = 0x37DDB3D7          # f32(1 / 37837.227237...)
NORMAL_CENTER = 131070                  # 4 * 32767.5
SINK_MULT = np.float32(20.0)            # position-0 keys of the prompt span
NOISE_MULT = np.float32(0.5)            # std of the ladder donors' perturbation

# Stream ids.
S_Q = 1            # (s, t, l, hq, c)   t in [0, T]
S_KSUF = 2         # (s, l, h, i, c)    i in [0, T)
S_VSUF = 3
S_KCLEAN = 4       # (p, l, h, j, c)
S_VCLEAN = 5
S_KFILL = 6        # (p, k, l, h, j, c) fresh filler of a donor slot
S_VFILL = 7
S_KNOISE = 8       # (p, k, l, h, j, c) perturbation of a ladder donor
S_VNOISE = 9
S_PMASK = 10       # (p, k, j)          which positions a ladder donor perturbs


def normal_scale() -> np.float32:
    return np.array([NORMAL_SCALE_BITS], dtype=np.uint32).view(np.float32)[0]


def q_mult(head_dim: int) -> np.float32:
    return np.float32(1.0 / np.sqrt(head_dim))


def mix(z: np.ndarray) -> np.ndarray:
    """splitmix64 finaliser on a uint64 array (wrapping arithmetic)."""
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * MIX1
        z = (z ^ (z >> np.uint64(27))) * MIX2
        return z ^ (z >> np.uint64(31))


def stream_state(seed: int, stream: int) -> np.uint64:
    with np.errstate(over="ignore"):
        x = np.array([(seed * 256 + stream) & 0xFFFFFFFFFFFFFFFF], dtype=np.uint64)
        return mix(x + GAMMA)[0]


def draw(seed: int, stream: int, idx: np.ndarray) -> np.ndarray:
    """uint64 output ``idx`` of stream (seed, stream)."""
    x0 = stream_state(seed, stream)
    idx = np.asarray(idx, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return mix(x0 + (idx + np.uint64(1)) * GAMMA)


def f32_to_bf16_rne(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (round to nearest, ties to even); finite inputs."""
    b = np.asarray(x, dtype=np.float32).view(np.uint32)
    r = ((b >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((b + r) >> np.uint32(16)).astype(np.uint16)


def bf16_to_f32(u: np.ndarray) -> np.ndarray:
    return (np.asarray(u, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def normal_f32(seed: int, stream: int, idx: np.ndarray) -> np.ndarray:
    """fp32 z of the definition above (before the multiplier and bf16 rounding)."""
    u = draw(seed, stream, idx)
    m = np.uint64(0xFFFF)
    c = ((u & m) + ((u >> np.uint64(16)) & m) + ((u >> np.uint64(32)) & m)
         + (u >> np.uint64(48))).astype(np.int64) - NORMAL_CENTER
    return (c.astype(np.float32) * normal_scale()).astype(np.float32)


def normal_bf16(seed: int, stream: int, idx: np.ndarray, mult=np.float32(1.0)) -> np.ndarray:
    z = normal_f32(seed, stream, idx)
    if np.ndim(mult) == 0 and np.float32(mult) == np.float32(1.0):
        return f32_to_bf16_rne(z)
    return f32_to_bf16_rne((z * np.asarray(mult, dtype=np.float32)).astype(np.float32))


def _lin(*coords_and_dims):
    """Row-major linear index of broadcastable coordinate arrays."""
    idx = np.uint64(0)
    for c, n in coords_and_dims:
        idx = idx * np.uint64(n) + np.asarray(c, dtype=np.uint64)
    return idx


class SynthInputs:
    """Regenerates any slice of a workload's inputs as bf16 bit patterns (uint16)."""

    def __init__(self, wl: W.Workload):
        self.wl = wl

    # -- per-sequence tensors -------------------------------------------------
    def q(self, s: int, t: int, l: int) -> np.ndarray:
        """Query of sequence s at step t, layer l: [Hq][d]."""
        wl = self.wl
        hq = np.arange(wl.num_q_heads)[:, None]
        c = np.arange(wl.head_dim)[None, :]
        idx = _lin((s, wl.num_sequences()), (t, wl.max_steps + 1), (l, wl.num_layers),
                   (hq, wl.num_q_heads), (c, wl.head_dim))
        return normal_bf16(wl.seed, S_Q, idx, q_mult(wl.head_dim))

    def suffix_kv(self, s: int, l: int, i0: int, i1: int):
        """Own generated-span K, V of sequence s, positions [i0, i1): [Hkv][n][d] each."""
        wl = self.wl
        h = np.arange(wl.num_kv_heads)[:, None, None]
        i = np.arange(i0, i1)[None, :, None]
        c = np.arange(wl.head_dim)[None, None, :]
        idx = _lin((s, wl.num_sequences()), (l, wl.num_layers), (h, wl.num_kv_heads),
                   (i, wl.max_steps), (c, wl.head_dim))
        return normal_bf16(wl.seed, S_KSUF, idx), normal_bf16(wl.seed, S_VSUF, idx)

    # -- prompt-span stores ---------------------------------------------------
    def _span_idx(self, p, l, j0, j1):
        wl = self.wl
        h = np.arange(wl.num_kv_heads)[:, None, None]
        j = np.arange(j0, j1)[None, :, None]
        c = np.arange(wl.head_dim)[None, None, :]
        return j, _lin((p, wl.num_prompts), (l, wl.num_layers), (h, wl.num_kv_heads),
                       (j, wl.prompt_len), (c, wl.head_dim))

    def clean_kv(self, p: int, l: int, j0: int = 0, j1: int | None = None):
        """Clean prompt-span K, V of prompt p at layer l, positions [j0, j1)."""
        wl = self.wl
        j1 = wl.prompt_len if j1 is None else j1
        j, idx = self._span_idx(p, l, j0, j1)
        kmult = np.where(j == 0, SINK_MULT, np.float32(1.0)).astype(np.float32)
        return (normal_bf16(wl.seed, S_KCLEAN, idx, kmult),
                normal_bf16(wl.seed, S_VCLEAN, idx))

    def perturbed(self, p: int, k: int, j: np.ndarray) -> np.ndarray:
        """Whether a ladder donor (slot k of prompt p) perturbs positions j."""
        wl = self.wl
        thr = W.PERTURB_THRESHOLD_24[wl.slot_kinds[k]]
        u = draw(wl.seed, S_PMASK, _lin((p, wl.num_prompts), (k, wl.num_donor_slots),
                                         (j, wl.prompt_len)))
        return (u >> np.uint64(40)) < np.uint64(thr)

    def donor_kv(self, p: int, k: int, l: int, j0: int = 0, j1: int | None = None):
        """Donor-slot K, V (slot k, a non-ZERO kind) of prompt p at layer l.

        BLANK and DIFF_FAMILY keep the template scaffold (first/last positions)
        of the clean span and hold fresh filler elsewhere; SAME_ALGO and
        DIFF_ALGO equal the clean span except at hashed non-scaffold positions,
        which carry clean + N(0, 0.5) noise.
        """
        wl = self.wl
        kind = wl.slot_kinds[k]
        if kind == W.ZERO:
            raise ValueError("ZERO donor slots are not stored")
        j1 = wl.prompt_len if j1 is None else j1
        ck, cv = self.clean_kv(p, l, j0, j1)
        jj = np.arange(j0, j1)
        scaffold = (jj < wl.scaffold_head) | (jj >= wl.prompt_len - wl.scaffold_tail)
        h = np.arange(wl.num_kv_heads)[:, None, None]
        j = jj[None, :, None]
        c = np.arange(wl.head_dim)[None, None, :]
        idx = _lin((p, wl.num_prompts), (k, wl.num_donor_slots), (l, wl.num_layers),
                   (h, wl.num_kv_heads), (j, wl.prompt_len), (c, wl.head_dim))
        if kind in (W.BLANK, W.DIFF_FAMILY):
            keep = scaffold[None, :, None]
            fk = normal_bf16(wl.seed, S_KFILL, idx)
            fv = normal_bf16(wl.seed, S_VFILL, idx)
            return np.where(keep, ck, fk), np.where(keep, cv, fv)
        pert = (~scaffold) & self.perturbed(p, k, jj)
        m = pert[None, :, None]
        nk = bf16_to_f32(normal_bf16(wl.seed, S_KNOISE, idx)) * NOISE_MULT
        nv = bf16_to_f32(normal_bf16(wl.seed, S_VNOISE, idx)) * NOISE_MULT
        pk = f32_to_bf16_rne((bf16_to_f32(ck) + nk).astype(np.float32))
        pv = f32_to_bf16_rne((bf16_to_f32(cv) + nv).astype(np.float32))
        return np.where(m, pk, ck), np.where(m, pv, cv)
