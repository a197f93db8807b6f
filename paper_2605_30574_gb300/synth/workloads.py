"""Synthetic sweep workloads shaped like the paper's models and prompts.

The paper (§2, §3) sweeps one splice intervention over a layer cutoff L, a
splice onset W and a donor kind (Table 1) on four chat models.  Its datasets
and weights are not available here, so every tensor is synthetic; this module
only fixes the *shapes* of those sweeps: model shape, prompt-span length T_p,
donor slots, decode steps T, the (L, W) grid, the scaffold extent of a
template-preserving donor, and how sweep cells are enumerated into sequences.

It holds none of the method's arithmetic (no splice rule, no attention); both
the CUDA path and the CPU oracle read their shapes from here.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Tuple

# Donor kinds of Table 1.  The integer values are the C ABI's
# ``splice_donor_kind`` values.
ZERO = 0
BLANK = 1
SAME_ALGO = 2
DIFF_ALGO = 3
DIFF_FAMILY = 4
KIND_NAMES = {ZERO: "ZERO", BLANK: "BLANK", SAME_ALGO: "SAME_ALGO",
              DIFF_ALGO: "DIFF_ALGO", DIFF_FAMILY: "DIFF_FAMILY"}

# Fraction of non-scaffold positions whose K/V are perturbed in the two
# within-family donors of the donor-noise ladder, as 24-bit thresholds on a
# per-position hash: round(p * 2**24) for p = 0.1 and p = 0.5.
PERTURB_THRESHOLD_24 = {SAME_ALGO: 1677722, DIFF_ALGO: 8388608}


@dataclass(frozen=True)
class Seq:
    """One sweep cell applied to one prompt: (prompt p, donor slot k, L, W)."""
    prompt: int
    slot: int
    L: int
    W: int


@dataclass(frozen=True)
class Workload:
    name: str
    num_layers: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    num_prompts: int
    prompt_len: int
    slot_kinds: Tuple[int, ...]
    max_steps: int
    L_values: Tuple[int, ...]
    W_values: Tuple[int, ...]
    scaffold_head: int
    scaffold_tail: int
    batch: int
    sliding_window: int = 0      # 0 = every layer attends to every key
    global_every: int = 0        # layer l is global iff (l + 1) % global_every == 0
    sm_scale: float = 1.0        # Q is pre-scaled by 1/sqrt(d) at generation
    seed: int = 0

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads

    @property
    def num_donor_slots(self) -> int:
        return len(self.slot_kinds)

    def is_scaffold(self, j: int) -> bool:
        return j < self.scaffold_head or j >= self.prompt_len - self.scaffold_tail

    def cells_per_prompt(self) -> int:
        return len(self.slot_kinds) * len(self.L_values) * len(self.W_values)

    def sequences(self) -> List[Seq]:
        """All sweep cells, prompt-major: prompt, then donor slot, then L, then W."""
        out = []
        for p in range(self.num_prompts):
            for k in range(len(self.slot_kinds)):
                for L in self.L_values:
                    for W in self.W_values:
                        out.append(Seq(p, k, L, W))
        return out

    def num_sequences(self) -> int:
        return self.num_prompts * self.cells_per_prompt()

    def num_batches(self) -> int:
        return -(-self.num_sequences() // self.batch)

    def batch_range(self, b: int) -> Tuple[int, int]:
        lo = b * self.batch
        return lo, min(lo + self.batch, self.num_sequences())

    def batch_prompts(self, b: int) -> Tuple[int, int]:
        """[first, last+1) of the prompts whose cells fall in batch b."""
        lo, hi = self.batch_range(b)
        c = self.cells_per_prompt()
        return lo // c, (hi - 1) // c + 1

    def layer_is_global(self, l: int) -> bool:
        if self.sliding_window <= 0:
            return True
        if self.global_every <= 0:
            return False
        return (l + 1) % self.global_every == 0


def _tiny() -> Workload:
    return Workload("tiny", 4, 8, 2, 64, 2, 128, (BLANK, ZERO), 16,
                    (0, 1, 2, 3, 4), (0, 4, 8, 16), 16, 8, batch=80)


def _qwen3_4b() -> Workload:
    return Workload("qwen3-4b", 36, 32, 8, 128, 8, 256, (BLANK, ZERO), 256,
                    tuple(range(0, 37, 4)), (0, 1, 2, 4, 8, 16, 32, 64), 24, 12,
                    batch=1280)


def _llama3_8b() -> Workload:
    return Workload("llama3-8b", 32, 32, 8, 128, 16, 512, (BLANK, ZERO), 512,
                    tuple(range(0, 33, 4)), (0, 2, 8, 32, 128), 24, 12, batch=1440)


def _gemma3_4b() -> Workload:
    return Workload("gemma3-4b", 34, 8, 4, 256, 8, 1024, (BLANK, ZERO), 256,
                    tuple(range(0, 35, 2)), (0, 4, 16, 64), 24, 12, batch=1152,
                    sliding_window=1024, global_every=6)


def _qwen3_8b_ladder() -> Workload:
    return Workload("qwen3-8b-ladder", 36, 32, 8, 128, 32, 4096,
                    (SAME_ALGO, DIFF_ALGO, DIFF_FAMILY, BLANK, ZERO), 1024,
                    (0, 9, 18, 27, 36), (0, 16, 64, 256), 24, 12, batch=512)


WORKLOADS = {w.name: w for w in (_tiny(), _qwen3_4b(), _llama3_8b(), _gemma3_4b(),
                                 _qwen3_8b_ladder())}
# Order of the five sweeps, smallest first.
WORKLOAD_ORDER = ("tiny", "qwen3-4b", "llama3-8b", "gemma3-4b", "qwen3-8b-ladder")


def get(name: str) -> Workload:
    return WORKLOADS[name]
