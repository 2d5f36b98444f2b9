"""ctypes loader for libcmc.so (the C ABI declared in include/cmc.h).

The shared library is built in-tree by `paper_2609_25537_gb300.build`.  When
it is missing, loading fails loudly: there is no fallback implementation.
"""

from __future__ import annotations

import ctypes
import os
import threading

PKG_DIR = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG_DIR, "libcmc.so")

# Every symbol include/cmc.h declares.
EXPORTS = (
    "cmc_status_string",
    "cmc_last_cuda_error",
    "cmc_denoise_workspace_size",
    "cmc_denoise",
    "cmc_bridge_epilogue",
    "cmc_score_select_workspace_size",
    "cmc_score_select",
    "cmc_question_select_workspace_size",
    "cmc_question_select",
    "cmc_window_append",
    "cmc_decode_attn_workspace_size",
    "cmc_two_tier_decode_attn",
    "cmc_decode_step",
    "cmc_decode_step_rope",
    "cmc_tier1_gather",
    "cmc_decode_attn_plan",
    "cmc_read_status",
    "cmc_set_l2_prefetch_tiles",
    "cmc_test_stall_attention_waits",
    "cmc_stage_copies",
    "cmc_score_select_static",
)

STATUS = {
    0: "CMC_OK",
    1: "CMC_ERR_NULL",
    2: "CMC_ERR_SHAPE",
    3: "CMC_ERR_RANGE",
    4: "CMC_ERR_ALIGN",
    5: "CMC_ERR_WORKSPACE",
    6: "CMC_ERR_CUDA",
}

DEVFLAG_BAD_INDEX = 1
DEVFLAG_BAD_POS = 2
DEVFLAG_TIMEOUT = 4


class CmcCopy(ctypes.Structure):
    """Mirror of `cmc_copy` (include/cmc.h)."""
    _fields_ = [("src", ctypes.c_void_p), ("dst", ctypes.c_void_p), ("bytes", ctypes.c_size_t)]


class CmcDims(ctypes.Structure):
    """Mirror of `cmc_dims` (include/cmc.h)."""
    _fields_ = [(name, ctypes.c_int32) for name in ("B", "L", "Hq", "Hkv", "d", "N", "k", "W")]

    def key(self):
        return tuple(getattr(self, f) for f, _ in self._fields_)


class CmcError(RuntimeError):
    def __init__(self, status: int, where: str, cuda_error: int = 0):
        self.status = status
        self.cuda_error = cuda_error
        msg = f"{where}: {STATUS.get(status, status)}"
        if cuda_error:
            msg += f" (cudaError {cuda_error})"
        super().__init__(msg)


_lib = None
_lock = threading.Lock()

_vp = ctypes.c_void_p
_i = ctypes.c_int
_sz = ctypes.c_size_t
_dims_p = ctypes.POINTER(CmcDims)

_SIGNATURES = {
    "cmc_status_string": (ctypes.c_char_p, [_i]),
    "cmc_last_cuda_error": (_i, []),
    "cmc_denoise_workspace_size": (_sz, [_i, _i]),
    "cmc_denoise": (_i, [_vp, _vp, _i, _i, _i, _i, ctypes.c_float, _i, _vp, _vp, _vp, _sz, _vp]),
    "cmc_bridge_epilogue": (_i, [_vp, _vp, _vp, ctypes.c_int64, _i, ctypes.c_float,
                                 ctypes.c_float, _vp, _vp]),
    "cmc_score_select_workspace_size": (_sz, [_i, _i]),
    "cmc_score_select": (_i, [_vp, _vp, _i, _i, _i, _i, _vp, _vp, _vp, _sz, _vp]),
    "cmc_question_select_workspace_size": (_sz, [_i, _i]),
    "cmc_question_select": (_i, [_vp, _vp, _i, _vp, _i, _i, _i, _i, _vp, _vp, _i, _vp, _vp, _vp,
                                 _vp, _vp, _sz, _vp]),
    "cmc_window_append": (_i, [_vp, _vp, _vp, _vp, _vp, _dims_p, _vp]),
    "cmc_decode_attn_workspace_size": (_sz, [_dims_p]),
    "cmc_two_tier_decode_attn": (_i, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _dims_p,
                                      ctypes.c_float, _vp, _vp, _sz, _vp]),
    "cmc_decode_step": (_i, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _dims_p,
                             ctypes.c_float, _vp, _vp, _sz, _vp]),
    "cmc_decode_step_rope": (_i, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _dims_p,
                                  ctypes.c_float, ctypes.c_double, ctypes.c_int64, _vp, _vp, _sz,
                                  _vp]),
    "cmc_tier1_gather": (_i, [_vp, _vp, _vp, _dims_p, _vp, _vp, _vp, _vp]),
    "cmc_decode_attn_plan": (_i, [_dims_p, _i, ctypes.POINTER(_i), ctypes.POINTER(_i)]),
    "cmc_read_status": (_i, [_vp, _i, ctypes.POINTER(ctypes.c_uint32), _vp]),
    "cmc_set_l2_prefetch_tiles": (_i, [_i]),
    "cmc_test_stall_attention_waits": (_i, [_i]),
    "cmc_stage_copies": (_i, [_vp, _i, _i, _vp]),
    "cmc_score_select_static": (_i, [_vp, _vp, _i, _i, _i, _i, _vp, _vp]),
}

# Largest B * N accepted by cmc_score_select_static (CMC_STATIC_SCORES_MAX).
STATIC_SCORES_MAX = 262144


def lib() -> ctypes.CDLL:
    """The loaded library.  Raises RuntimeError when it has not been built."""
    global _lib
    if _lib is None:
        with _lock:
            if _lib is None:
                if not os.path.exists(LIB_PATH):
                    raise RuntimeError(
                        f"libcmc.so not found at {LIB_PATH}: build it first "
                        "(python -c 'import __graft_entry__ as g; g.build()')")
                handle = ctypes.CDLL(LIB_PATH)
                for name, (res, args) in _SIGNATURES.items():
                    fn = getattr(handle, name)
                    fn.restype = res
                    fn.argtypes = args
                _lib = handle
    return _lib


def check(status: int, where: str) -> None:
    if status != 0:
        cuda_err = lib().cmc_last_cuda_error() if status == 6 else 0
        raise CmcError(status, where, cuda_err)
