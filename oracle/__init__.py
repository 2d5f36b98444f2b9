"""CPU fp64 oracle of the CMC two-tier decode path (test infrastructure).

This package is test infrastructure, not part of the product: only the tests,
`__graft_entry__.smoke()` and the CPU-baseline / reference legs of `bench.py`
import it.  It shares no code with the CUDA library; the only thing both sides
share is the seeded input generator in `workloads/`.
"""

from .cmc_oracle import (
    bf16_to_f64,
    cosine_scores,
    select_top_k,
    score_select,
    denoise_pass,
    keep_minimum,
    denoise_keep,
    denoise,
    bridge_epilogue,
    question_vector,
    tier2_start,
    cme_locate,
    question_select,
    window_append,
    window_slots,
    softmax_attention,
    two_tier_kv,
    two_tier_attention_head,
    two_tier_attention,
    decode_step,
    default_scale,
    rope_angles,
    rope_rotate,
    f64_to_bf16_bits,
    decode_step_rope,
)

__all__ = [
    "bf16_to_f64",
    "cosine_scores",
    "select_top_k",
    "score_select",
    "denoise_pass",
    "keep_minimum",
    "denoise_keep",
    "denoise",
    "bridge_epilogue",
    "question_vector",
    "tier2_start",
    "cme_locate",
    "question_select",
    "window_append",
    "window_slots",
    "softmax_attention",
    "two_tier_kv",
    "two_tier_attention_head",
    "two_tier_attention",
    "decode_step",
    "default_scale",
    "rope_angles",
    "rope_rotate",
    "f64_to_bf16_bits",
    "decode_step_rope",
]
