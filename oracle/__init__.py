"""CPU fp64 oracle for the spliced decode-attention path.

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and ``bench.py``'s CPU-baseline / reference legs, never by the product path.
See ``splice_oracle`` for what it computes and how it is pinned.
"""
from .splice_oracle import (SRC_CLEAN, SRC_ZERO, SRC_DONOR0, splice_source,  # noqa: F401
                            visible_range, layer_is_global, bf16_to_f64,
                            spliced_prompt_kv, attend, decode_attn, partial,
                            merge_partials, delta_positions, delta_encode, delta_decode,
                            pack_mask_words)
