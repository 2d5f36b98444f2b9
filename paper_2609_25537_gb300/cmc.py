"""Python binding of libcmc: the CMC two-tier decode path on GB300.

Argument marshalling only.  Each function checks the tensors it is given
(device, dtype, contiguity, shapes), derives the sizes, and calls the C ABI
with raw device pointers and the current torch CUDA stream.  Every step of the
computation runs in the library's CUDA kernels; there is no CPU path.

Tensor layouts (row-major, last index fastest):

  question_emb  fp32 [B, D]            cme_bank  fp32 [B, N, D]
  q             bf16 [B, L, Hq, d]     out       bf16 [B, L, Hq, d]
  tier1_k/v     bf16 [B, L, Hkv, N, d] idx       int32 [B, k]
  ring_k/v      bf16 [B, L, Hkv, W, d] pos       int64 [B]
  k_new/v_new   bf16 [B, L, Hkv, d]

Tier-1 selection in the attention calls: an ``idx`` tensor [B, k] gathers
rows of the bank by index at every step; ``idx=None`` takes every row of
``tier1_k``/``tier1_v`` in order (k = N), which is how the dense Tier-1 cache
made once per question by :func:`tier1_gather` is passed.
"""

from __future__ import annotations

import ctypes
import functools
import os
from typing import Dict, Optional, Tuple

import torch

from ._lib import CmcCopy, CmcDims, check, lib, DEVFLAG_BAD_INDEX, DEVFLAG_BAD_POS, DEVFLAG_TIMEOUT

__all__ = [
    "CmcDims",
    "DecodeWorkspace",
    "denoise",
    "bridge_epilogue",
    "score_select",
    "score_select_workspace_size",
    "question_select",
    "window_append",
    "two_tier_decode_attn",
    "decode_step",
    "tier1_gather",
    "decode_attn_workspace_size",
    "decode_attn_plan",
    "set_l2_prefetch_tiles",
    "dims_of",
    "stage_copies",
    "DEVFLAG_BAD_INDEX",
    "DEVFLAG_BAD_POS",
    "DEVFLAG_TIMEOUT",
]


# With CMC_NVTX set (not "0") when the module is imported, every device call
# below is wrapped in an NVTX range named after it ("cmc.decode_step", ...),
# for profiler timelines; otherwise the functions are left as they are.
_NVTX = os.environ.get("CMC_NVTX", "") not in ("", "0")


def _ranged(fn):
    if not _NVTX:
        return fn
    name = "cmc." + fn.__name__

    @functools.wraps(fn)
    def wrapped(*args, **kwargs):
        torch.cuda.nvtx.range_push(name)
        try:
            return fn(*args, **kwargs)
        finally:
            torch.cuda.nvtx.range_pop()
    return wrapped


def _p(t: Optional[torch.Tensor]) -> ctypes.c_void_p:
    return ctypes.c_void_p(0 if t is None else t.data_ptr())


def _stream(device: torch.device) -> ctypes.c_void_p:
    return ctypes.c_void_p(torch.cuda.current_stream(device).cuda_stream)


def _need(t: torch.Tensor, name: str, dtype: torch.dtype, ndim: int, device=None) -> None:
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor (the library has no CPU path)")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if t.dim() != ndim:
        raise ValueError(f"{name} must have {ndim} dims, got shape {tuple(t.shape)}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if device is not None and t.device != device:
        raise ValueError(f"{name} is on {t.device}, expected {device}")


# ----------------------------------------------------------------------------
# Graph-based context denoising
# ----------------------------------------------------------------------------

@_ranged
def denoise(emb: torch.Tensor, *, n_tokens: Optional[torch.Tensor] = None, g: int = 3,
            tau: float = 0.05, keep_every: int = 16,
            workspace: Optional[torch.Tensor] = None) -> Tuple[torch.Tensor, torch.Tensor]:
    """Positions of the tokens kept by the graph-based denoising, int32
    [B, n_max] ascending then -1, and their counts int32 [B]; see
    cmc_denoise.  Defaults: the paper's g = 3, tau = 0.05, keep-minimum 16.
    A given ``workspace`` must have been zero-filled before its first use."""
    _need(emb, "emb", torch.float32, 3)
    dev = emb.device
    B, n_max, H = emb.shape
    if n_tokens is not None:
        _need(n_tokens, "n_tokens", torch.int32, 1, dev)
        if int(n_tokens.shape[0]) != B:
            raise ValueError("n_tokens must be [B]")
    kept = torch.empty((B, n_max), dtype=torch.int32, device=dev)
    count = torch.empty(B, dtype=torch.int32, device=dev)
    need = int(lib().cmc_denoise_workspace_size(B, n_max))
    if workspace is None:
        workspace = _counter_workspace("denoise", need, dev)
    st = lib().cmc_denoise(_p(emb), _p(n_tokens), B, n_max, H, g, float(tau), keep_every,
                           _p(kept), _p(count), _p(workspace),
                           workspace.numel() * workspace.element_size(), _stream(dev))
    check(st, "cmc_denoise")
    return kept, count


# ----------------------------------------------------------------------------
# MemoryBridge output
# ----------------------------------------------------------------------------

@_ranged
def bridge_epilogue(x: torch.Tensor, nu: float, *, gamma: Optional[torch.Tensor] = None,
                    beta: Optional[torch.Tensor] = None, eps: float = 1e-5,
                    out: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Decoder-ready CMEs from the MemoryBridge MLP output x (fp32 [..., D]):
    LayerNorm, nu tanh, and the 2 nu norm cap; see cmc_bridge_epilogue."""
    _need(x, "x", torch.float32, x.dim())
    dev = x.device
    D = int(x.shape[-1])
    rows = x.numel() // D if D else 0
    for t, name in ((gamma, "gamma"), (beta, "beta")):
        if t is not None:
            _need(t, name, torch.float32, 1, dev)
            if int(t.shape[0]) != D:
                raise ValueError(f"{name} must be [{D}]")
    if out is None:
        out = torch.empty_like(x)
    _need(out, "out", torch.float32, x.dim(), dev)
    if out.shape != x.shape:
        raise ValueError("out must have the shape of x")
    st = lib().cmc_bridge_epilogue(_p(x), _p(gamma), _p(beta), rows, D, float(eps), float(nu),
                                   _p(out), _stream(dev))
    check(st, "cmc_bridge_epilogue")
    return out


# ----------------------------------------------------------------------------
# Tier-1: scoring and selection
# ----------------------------------------------------------------------------

def score_select_workspace_size(B: int, N: int) -> int:
    return int(lib().cmc_score_select_workspace_size(B, N))


_counter_ws_cache: Dict[Tuple, torch.Tensor] = {}


def _counter_workspace(kind: str, nbytes: int, device: torch.device) -> torch.Tensor:
    """A zero-filled workspace, one per (kind, device, stream, size): its
    completion counters start at zero, and every call leaves them so."""
    key = (kind, device.index, torch.cuda.current_stream(device).cuda_stream, nbytes)
    ws = _counter_ws_cache.get(key)
    if ws is None:
        ws = torch.zeros(nbytes, dtype=torch.uint8, device=device)
        _counter_ws_cache[key] = ws
    return ws


@_ranged
def score_select(question_emb: torch.Tensor, cme_bank: torch.Tensor, k: int, *,
                 idx_out: Optional[torch.Tensor] = None,
                 scores_out: Optional[torch.Tensor] = None,
                 workspace: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Top-k CMEs by cosine similarity to the question vector, as int32 [B, k]
    indices in ascending (document) order.  See cmc_score_select.  A given
    ``workspace`` must have been zero-filled before its first use."""
    _need(cme_bank, "cme_bank", torch.float32, 3)
    dev = cme_bank.device
    _need(question_emb, "question_emb", torch.float32, 2, dev)
    B, N, D = cme_bank.shape
    if tuple(question_emb.shape) != (B, D):
        raise ValueError(f"question_emb shape {tuple(question_emb.shape)} != {(B, D)}")
    if idx_out is None:
        idx_out = torch.empty((B, k), dtype=torch.int32, device=dev)
    _need(idx_out, "idx_out", torch.int32, 2, dev)
    if tuple(idx_out.shape) != (B, k):
        raise ValueError(f"idx_out shape {tuple(idx_out.shape)} != {(B, k)}")
    if scores_out is not None:
        _need(scores_out, "scores_out", torch.float32, 2, dev)
        if tuple(scores_out.shape) != (B, N):
            raise ValueError(f"scores_out shape {tuple(scores_out.shape)} != {(B, N)}")
    if workspace is None:
        workspace = _counter_workspace("select", score_select_workspace_size(B, N), dev)
    ws_bytes = workspace.numel() * workspace.element_size()
    st = lib().cmc_score_select(_p(question_emb), _p(cme_bank), B, N, D, k, _p(idx_out),
                                _p(scores_out), _p(workspace), ws_bytes, _stream(dev))
    check(st, "cmc_score_select")
    return idx_out


@_ranged
def question_select(question_tokens: torch.Tensor, cme_bank: torch.Tensor, k: int, *,
                    q_len: Optional[torch.Tensor] = None,
                    chunk_offset: Optional[torch.Tensor] = None,
                    ctx_len: Optional[torch.Tensor] = None, W: Optional[int] = None,
                    workspace: Optional[torch.Tensor] = None):
    """The question-side prologue; see cmc_question_select.  Returns
    (q_vec fp32 [B, D], idx int32 [B, k], alpha int32 [B] or None,
    start int32 [B] or None); alpha and start when chunk_offset, ctx_len
    and W are given."""
    _need(cme_bank, "cme_bank", torch.float32, 3)
    dev = cme_bank.device
    _need(question_tokens, "question_tokens", torch.float32, 3, dev)
    B, N, D = cme_bank.shape
    Bq, Lq, Dq = question_tokens.shape
    if (Bq, Dq) != (B, D):
        raise ValueError(f"question_tokens shape {tuple(question_tokens.shape)} != ({B}, Lq, {D})")
    if q_len is not None:
        _need(q_len, "q_len", torch.int32, 1, dev)
        if int(q_len.shape[0]) != B:
            raise ValueError("q_len must be [B]")
    locate = chunk_offset is not None
    if locate:
        _need(chunk_offset, "chunk_offset", torch.int32, 2, dev)
        _need(ctx_len, "ctx_len", torch.int32, 1, dev)
        if tuple(chunk_offset.shape) != (B, N) or int(ctx_len.shape[0]) != B or W is None:
            raise ValueError("chunk_offset [B, N], ctx_len [B] and W are needed together")
    q_vec = torch.empty((B, D), dtype=torch.float32, device=dev)
    idx = torch.empty((B, k), dtype=torch.int32, device=dev)
    alpha = torch.empty(B, dtype=torch.int32, device=dev) if locate else None
    start = torch.empty(B, dtype=torch.int32, device=dev) if locate else None
    need = int(lib().cmc_question_select_workspace_size(B, N))
    if workspace is None:
        workspace = _counter_workspace("question", need, dev)
    st = lib().cmc_question_select(
        _p(question_tokens), _p(q_len), Lq, _p(cme_bank), B, N, D, k, _p(chunk_offset),
        _p(ctx_len), int(W or 0), _p(q_vec), _p(idx), _p(alpha), _p(start), _p(workspace),
        workspace.numel() * workspace.element_size(), _stream(dev))
    check(st, "cmc_question_select")
    return q_vec, idx, alpha, start


# ----------------------------------------------------------------------------
# Decode attention
# ----------------------------------------------------------------------------

def dims_of(q: torch.Tensor, tier1_k: torch.Tensor, idx: Optional[torch.Tensor],
            ring_k: torch.Tensor) -> CmcDims:
    B, L, Hq, d = q.shape
    Bk, Lk, Hkv, N, dk = tier1_k.shape
    Br, Lr, Hr, W, dr = ring_k.shape
    k = N if idx is None else int(idx.shape[1])
    if (Bk, Lk, dk) != (B, L, d) or (Br, Lr, Hr, dr) != (B, L, Hkv, d):
        raise ValueError(f"inconsistent shapes: q {tuple(q.shape)}, tier1 {tuple(tier1_k.shape)}, "
                         f"ring {tuple(ring_k.shape)}")
    if idx is not None and int(idx.shape[0]) != B:
        raise ValueError(f"idx shape {tuple(idx.shape)} does not match batch {B}")
    return CmcDims(B, L, Hq, Hkv, d, N, k, W)


def decode_attn_workspace_size(dims: CmcDims) -> int:
    return int(lib().cmc_decode_attn_workspace_size(ctypes.byref(dims)))


def decode_attn_plan(dims: CmcDims, fused: bool = True, rope: bool = False) -> Tuple[int, int]:
    """(grid size, kernel launches per call) of the attention entry points for
    `dims` on the current device; see cmc_decode_attn_plan."""
    ctas, launches = ctypes.c_int(0), ctypes.c_int(0)
    mode = 2 if rope else (1 if fused else 0)
    st = lib().cmc_decode_attn_plan(ctypes.byref(dims), mode, ctypes.byref(ctas),
                                    ctypes.byref(launches))
    check(st, "cmc_decode_attn_plan")
    return int(ctas.value), int(launches.value)


class DecodeWorkspace:
    """Zero-filled device workspace for the attention entry points.

    Holds the device status word and the fp32 partial results of keys split
    between CTAs.  Calls sharing one workspace must be ordered on one stream."""

    def __init__(self, dims: CmcDims, device: torch.device):
        n = decode_attn_workspace_size(dims)
        if n == 0:
            raise ValueError(f"unsupported dims {dims.key()}")
        self.dims = dims
        self.nbytes = n
        self.buf = torch.zeros(n, dtype=torch.uint8, device=device)

    def status(self, clear: bool = True) -> int:
        """CMC_DEVFLAG_* bits raised by kernels since the last clear (synchronises)."""
        flags = ctypes.c_uint32(0)
        st = lib().cmc_read_status(_p(self.buf), 1 if clear else 0, ctypes.byref(flags),
                                   _stream(self.buf.device))
        check(st, "cmc_read_status")
        return int(flags.value)


_ws_cache: Dict[Tuple, DecodeWorkspace] = {}


def _workspace_for(dims: CmcDims, device: torch.device) -> DecodeWorkspace:
    key = (device.index, torch.cuda.current_stream(device).cuda_stream, dims.key())
    ws = _ws_cache.get(key)
    if ws is None:
        ws = DecodeWorkspace(dims, device)
        _ws_cache[key] = ws
    return ws


def _attn_args(q, tier1_k, tier1_v, idx, ring_k, ring_v, pos, out):
    _need(q, "q", torch.bfloat16, 4)
    dev = q.device
    _need(tier1_k, "tier1_k", torch.bfloat16, 5, dev)
    _need(tier1_v, "tier1_v", torch.bfloat16, 5, dev)
    _need(ring_k, "ring_k", torch.bfloat16, 5, dev)
    _need(ring_v, "ring_v", torch.bfloat16, 5, dev)
    _need(pos, "pos", torch.int64, 1, dev)
    if idx is not None:
        _need(idx, "idx", torch.int32, 2, dev)
    if tier1_v.shape != tier1_k.shape or ring_v.shape != ring_k.shape:
        raise ValueError("K and V tensors must have the same shapes")
    dims = dims_of(q, tier1_k, idx, ring_k)
    if int(pos.shape[0]) != dims.B:
        raise ValueError(f"pos shape {tuple(pos.shape)} does not match batch {dims.B}")
    if out is None:
        out = torch.empty_like(q)
    _need(out, "out", torch.bfloat16, 4, dev)
    if out.shape != q.shape:
        raise ValueError("out must have the shape of q")
    return dims, dev, out


def _scale(scale: Optional[float]) -> float:
    return 0.0 if scale is None else float(scale)


@_ranged
def two_tier_decode_attn(q, tier1_k, tier1_v, idx, ring_k, ring_v, pos, *,
                         scale: Optional[float] = None, out: Optional[torch.Tensor] = None,
                         workspace: Optional[DecodeWorkspace] = None) -> torch.Tensor:
    """Decode attention over [Tier-1 rows at idx | occupied ring slots]; see
    cmc_two_tier_decode_attn.  Returns bf16 [B, L, Hq, d]."""
    dims, dev, out = _attn_args(q, tier1_k, tier1_v, idx, ring_k, ring_v, pos, out)
    ws = workspace if workspace is not None else _workspace_for(dims, dev)
    st = lib().cmc_two_tier_decode_attn(
        _p(q), _p(tier1_k), _p(tier1_v), _p(idx), _p(ring_k), _p(ring_v), _p(pos),
        ctypes.byref(dims), _scale(scale), _p(out), _p(ws.buf), ws.nbytes, _stream(dev))
    check(st, "cmc_two_tier_decode_attn")
    return out


@_ranged
def decode_step(q, tier1_k, tier1_v, idx, ring_k, ring_v, pos, k_new, v_new, *,
                scale: Optional[float] = None, out: Optional[torch.Tensor] = None,
                workspace: Optional[DecodeWorkspace] = None,
                rope_theta: Optional[float] = None, rope_offset: int = 0) -> torch.Tensor:
    """Fused decode step: append (k_new, v_new) to the ring, then attend; see
    cmc_decode_step.  Updates ring_k, ring_v and pos in place.

    With ``rope_theta`` the step is that of a real GQA layer (see
    cmc_decode_step_rope): q and k_new are given before rotary embedding and
    are rotated at position ``rope_offset + pos[b]`` inside the launch."""
    dims, dev, out = _attn_args(q, tier1_k, tier1_v, idx, ring_k, ring_v, pos, out)
    _need(k_new, "k_new", torch.bfloat16, 4, dev)
    _need(v_new, "v_new", torch.bfloat16, 4, dev)
    want = (dims.B, dims.L, dims.Hkv, dims.d)
    if tuple(k_new.shape) != want or tuple(v_new.shape) != want:
        raise ValueError(f"k_new/v_new must be {want}")
    ws = workspace if workspace is not None else _workspace_for(dims, dev)
    if rope_theta is None:
        st = lib().cmc_decode_step(
            _p(q), _p(tier1_k), _p(tier1_v), _p(idx), _p(ring_k), _p(ring_v), _p(pos),
            _p(k_new), _p(v_new), ctypes.byref(dims), _scale(scale), _p(out), _p(ws.buf),
            ws.nbytes, _stream(dev))
        check(st, "cmc_decode_step")
    else:
        st = lib().cmc_decode_step_rope(
            _p(q), _p(tier1_k), _p(tier1_v), _p(idx), _p(ring_k), _p(ring_v), _p(pos),
            _p(k_new), _p(v_new), ctypes.byref(dims), _scale(scale), float(rope_theta),
            int(rope_offset), _p(out), _p(ws.buf), ws.nbytes, _stream(dev))
        check(st, "cmc_decode_step_rope")
    return out


def set_l2_prefetch_tiles(tiles: int) -> None:
    """Box tiles per CTA the attention launches made afterwards prefetch into
    L2 before their grid dependency wait (a hint); see
    cmc_set_l2_prefetch_tiles.  Default 5 (one stream of launches); 0 suits
    several streams of independent requests' launches."""
    check(lib().cmc_set_l2_prefetch_tiles(int(tiles)), "cmc_set_l2_prefetch_tiles")


@_ranged
def tier1_gather(bank_k: torch.Tensor, bank_v: torch.Tensor, idx: torch.Tensor, *,
                 out_k: Optional[torch.Tensor] = None, out_v: Optional[torch.Tensor] = None,
                 workspace: Optional[DecodeWorkspace] = None
                 ) -> Tuple[torch.Tensor, torch.Tensor]:
    """Dense Tier-1 cache of the selected rows, bf16 [B, L, Hkv, k, d] each for
    K and V; see cmc_tier1_gather.  Out-of-range indices raise
    DEVFLAG_BAD_INDEX in ``workspace``'s status word when one is given."""
    _need(bank_k, "bank_k", torch.bfloat16, 5)
    dev = bank_k.device
    _need(bank_v, "bank_v", torch.bfloat16, 5, dev)
    _need(idx, "idx", torch.int32, 2, dev)
    if bank_v.shape != bank_k.shape:
        raise ValueError("bank_v must have the shape of bank_k")
    B, L, Hkv, N, d = bank_k.shape
    k = int(idx.shape[1])
    if int(idx.shape[0]) != B:
        raise ValueError(f"idx shape {tuple(idx.shape)} does not match batch {B}")
    want = (B, L, Hkv, k, d)
    if out_k is None:
        out_k = torch.empty(want, dtype=torch.bfloat16, device=dev)
    if out_v is None:
        out_v = torch.empty(want, dtype=torch.bfloat16, device=dev)
    for t, name in ((out_k, "out_k"), (out_v, "out_v")):
        _need(t, name, torch.bfloat16, 5, dev)
        if tuple(t.shape) != want:
            raise ValueError(f"{name} must be {want}")
    dims = CmcDims(B, L, Hkv, Hkv, d, N, k, 1)
    status = None if workspace is None else workspace.buf
    st = lib().cmc_tier1_gather(_p(bank_k), _p(bank_v), _p(idx), ctypes.byref(dims), _p(out_k),
                                _p(out_v), _p(status), _stream(dev))
    check(st, "cmc_tier1_gather")
    return out_k, out_v


@_ranged
def window_append(ring_k: torch.Tensor, ring_v: torch.Tensor, pos: torch.Tensor,
                  k_new: torch.Tensor, v_new: torch.Tensor) -> None:
    """Append one token per sequence to the Tier-2 ring; see cmc_window_append."""
    _need(ring_k, "ring_k", torch.bfloat16, 5)
    dev = ring_k.device
    _need(ring_v, "ring_v", torch.bfloat16, 5, dev)
    _need(pos, "pos", torch.int64, 1, dev)
    _need(k_new, "k_new", torch.bfloat16, 4, dev)
    _need(v_new, "v_new", torch.bfloat16, 4, dev)
    B, L, Hkv, W, d = ring_k.shape
    if ring_v.shape != ring_k.shape:
        raise ValueError("ring_v must have the shape of ring_k")
    if tuple(k_new.shape) != (B, L, Hkv, d) or tuple(v_new.shape) != (B, L, Hkv, d):
        raise ValueError(f"k_new/v_new must be {(B, L, Hkv, d)}")
    if int(pos.shape[0]) != B:
        raise ValueError("pos must be [B]")
    dims = CmcDims(B, L, Hkv, Hkv, d, 1, 0, W)
    st = lib().cmc_window_append(_p(ring_k), _p(ring_v), _p(pos), _p(k_new), _p(v_new),
                                 ctypes.byref(dims), _stream(dev))
    check(st, "cmc_window_append")


# ----------------------------------------------------------------------------
# Staging copies (host <-> device traffic of a decode loop)
# ----------------------------------------------------------------------------

@_ranged
def stage_copies(pairs, *, wait_first: bool = False, device: Optional[torch.device] = None) -> None:
    """Copy each (src, dst) tensor pair, byte for byte, in one kernel launch on
    the current stream; see cmc_stage_copies.  Host tensors must be pinned
    (their memory is then mapped for the device).  With wait_first=False the
    copies overlap the kernel before the call on the stream (the caller keeps
    that kernel off every source and destination) and the launch completes
    after it."""
    pairs = list(pairs)
    if len(pairs) > 4:
        raise ValueError("at most 4 copies per call")
    arr = (CmcCopy * max(1, len(pairs)))()
    dev = device
    for i, (src, dst) in enumerate(pairs):
        for t, name in ((src, "src"), (dst, "dst")):
            if not isinstance(t, torch.Tensor) or not t.is_contiguous():
                raise ValueError(f"{name} must be a contiguous tensor")
            if not t.is_cuda and not t.is_pinned():
                raise ValueError(f"{name} must be a CUDA tensor or pinned host memory")
            if t.is_cuda:
                if dev is None:
                    dev = t.device
                elif t.device != dev:
                    raise ValueError("all device tensors must be on one device")
        nb = src.numel() * src.element_size()
        if dst.numel() * dst.element_size() != nb:
            raise ValueError("src and dst sizes differ")
        arr[i].src = src.data_ptr()
        arr[i].dst = dst.data_ptr()
        arr[i].bytes = nb
    if dev is None:
        dev = torch.device("cuda", torch.cuda.current_device())
    st = lib().cmc_stage_copies(ctypes.cast(arr, ctypes.c_void_p), len(pairs),
                                1 if wait_first else 0, _stream(dev))
    check(st, "cmc_stage_copies")
