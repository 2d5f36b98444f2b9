"""CMC two-tier KV-cache decode path for GB300 (sm_103a).

Question-guided top-K selection of Context Memory Embeddings (Tier-1), a
local-window ring (Tier-2) and GQA decode attention over [Tier-1 | Tier-2],
as hand-written CUDA kernels behind the C ABI of include/cmc.h.
"""

from .cmc import (  # noqa: F401
    CmcDims,
    DecodeWorkspace,
    DEVFLAG_BAD_INDEX,
    DEVFLAG_BAD_POS,
    DEVFLAG_TIMEOUT,
    bridge_epilogue,
    decode_attn_plan,
    decode_attn_workspace_size,
    decode_step,
    denoise,
    dims_of,
    question_select,
    score_select,
    score_select_workspace_size,
    set_l2_prefetch_tiles,
    stage_copies,
    tier1_gather,
    two_tier_decode_attn,
    window_append,
)
from ._lib import CmcError, EXPORTS, LIB_PATH, lib  # noqa: F401
