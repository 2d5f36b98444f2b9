"""The C ABI on the host: the library builds, loads and exports every symbol
include/cmc.h declares; argument checks fail with the documented status
before any CUDA call; workspace-size queries follow their formulas.  None of
these tests launches a kernel, so they run without a GPU."""

import ctypes
import os
import re

import pytest

import paper_2609_25537_gb300 as cmc
from paper_2609_25537_gb300 import _lib
from paper_2609_25537_gb300.build import build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "cmc.h")

OK, NULL, SHAPE, RANGE, ALIGN, WORKSPACE = 0, 1, 2, 3, 4, 5


@pytest.fixture(scope="module")
def L():
    build()
    return cmc.lib()


def _declared():
    src = open(HEADER).read()
    return re.findall(r"CMC_API\s+[\w\s\*]+?\b(cmc_\w+)\s*\(", src)


def test_header_and_binding_agree():
    names = _declared()
    assert len(names) == len(set(names)) and names
    assert set(names) == set(_lib.EXPORTS)


def test_library_exports_every_declared_symbol(L):
    for name in _declared():
        assert hasattr(L, name), name


def test_status_strings(L):
    for code in range(7):
        s = L.cmc_status_string(code).decode()
        assert s.startswith(_lib.STATUS[code])
    assert L.cmc_last_cuda_error() == 0


FAKE = 0x10000  # 16-byte aligned, never dereferenced: these calls fail before any launch

# The fake-pointer checks run only where no GPU is visible, so that a bug in
# the argument checks can never launch a kernel on fake pointers.
import torch  # noqa: E402

host_only = pytest.mark.skipif(torch.cuda.is_available(),
                               reason="fake-pointer argument checks run only without a GPU")


def _sel(L, qe=FAKE, bank=FAKE, B=2, N=64, D=16, k=8, idx=FAKE, scores=0, ws=FAKE, wsb=1 << 20):
    return L.cmc_score_select(qe, bank, B, N, D, k, idx, scores, ws, wsb, None)


@host_only
def test_score_select_argument_checks(L):
    assert _sel(L, B=0) == SHAPE
    assert _sel(L, N=0) == SHAPE
    assert _sel(L, D=6) == SHAPE
    assert _sel(L, D=0) == SHAPE
    assert _sel(L, k=65) == RANGE
    assert _sel(L, k=-1) == RANGE
    assert _sel(L, qe=0) == NULL
    assert _sel(L, bank=0) == NULL
    assert _sel(L, idx=0) == NULL
    assert _sel(L, bank=FAKE + 4) == ALIGN
    assert _sel(L, ws=0) == WORKSPACE
    assert _sel(L, wsb=2 * 64 * 4 - 1) == WORKSPACE
    assert _sel(L, wsb=512 + 255) == WORKSPACE  # room for the scores, not the counters
    assert _sel(L, ws=0, scores=FAKE, wsb=0, bank=FAKE + 4) == ALIGN  # no workspace: scores_out


def test_score_select_workspace_size(L):
    # 1200 bytes of scores rounded up to 256, 3 counters rounded up to 256,
    # then 3 histograms of 2,048 counts
    assert L.cmc_score_select_workspace_size(3, 100) == 1280 + 256 + 3 * 8192
    assert L.cmc_score_select_workspace_size(0, 100) == 0


def _dims(**kw):
    base = dict(B=2, L=3, Hq=8, Hkv=2, d=128, N=100, k=10, W=16)
    base.update(kw)
    return cmc.CmcDims(*(base[f] for f, _ in cmc.CmcDims._fields_))


def _attn(L, dims, q=FAKE, idx=FAKE, ws=FAKE, wsb=1 << 30, out=FAKE, pos=FAKE):
    return L.cmc_two_tier_decode_attn(q, FAKE, FAKE, idx, FAKE, FAKE, pos, ctypes.byref(dims),
                                      0.0, out, ws, wsb, None)


def _step(L, dims, k_new=FAKE, ws=FAKE, wsb=1 << 30):
    return L.cmc_decode_step(FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, k_new, FAKE,
                             ctypes.byref(dims), 0.0, FAKE, ws, wsb, None)


@host_only
def test_attention_argument_checks(L):
    assert _attn(L, _dims(d=96)) == SHAPE
    assert _attn(L, _dims(Hq=6)) == SHAPE          # Hq % Hkv != 0
    assert _attn(L, _dims(Hq=32, Hkv=2)) == SHAPE  # G = 16 unsupported
    assert _attn(L, _dims(B=0)) == SHAPE
    assert _attn(L, _dims(W=0)) == SHAPE
    assert _attn(L, _dims(k=101)) == RANGE
    assert _attn(L, _dims(k=-1)) == RANGE
    assert _attn(L, _dims(), q=0) == NULL
    # idx NULL is identity selection (Tier-1 = rows 0 .. k-1): not an error
    assert _attn(L, _dims(), idx=0) not in (NULL, SHAPE, RANGE, ALIGN, WORKSPACE)
    assert _attn(L, _dims(), out=0) == NULL
    assert _attn(L, _dims(), q=FAKE + 2) == ALIGN
    assert _attn(L, _dims(), pos=FAKE + 4) == ALIGN
    assert _attn(L, _dims(), ws=0) == WORKSPACE
    assert _attn(L, _dims(), wsb=16) == WORKSPACE
    assert _step(L, _dims(), k_new=0) == NULL
    assert _step(L, _dims(), k_new=FAKE + 8) == ALIGN
    assert _step(L, _dims(), wsb=16) == WORKSPACE
    assert L.cmc_two_tier_decode_attn(FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None, 0.0, FAKE,
                                      FAKE, 1 << 30, None) == NULL


@host_only
def test_window_append_argument_checks(L):
    d = _dims()
    assert L.cmc_window_append(0, FAKE, FAKE, FAKE, FAKE, ctypes.byref(d), None) == NULL
    assert L.cmc_window_append(FAKE, FAKE, FAKE + 4, FAKE, FAKE, ctypes.byref(d), None) == ALIGN
    assert L.cmc_window_append(FAKE, FAKE, FAKE, FAKE, FAKE, ctypes.byref(_dims(d=32)),
                               None) == SHAPE


def test_attention_workspace_size(L):
    # a 256-byte status header, 8 bytes per sequence padded to 256, then one
    # fp32 partial record per (unit, 64-key tile) slot: max and sum per head
    # (2G floats, padded to a multiple of 4) and the output, G * d floats;
    # a unit has ceil(k / 64) Tier-1 tiles and ceil(W / 64) ring tiles
    d = _dims()
    units = 2 * 3 * 2
    G = 4
    n = L.cmc_decode_attn_workspace_size(ctypes.byref(d))
    assert n == 256 + 256 + units * (1 + 1) * G * (128 + 2) * 4
    big = _dims(k=100, W=1000)
    assert L.cmc_decode_attn_workspace_size(ctypes.byref(big)) == (
        256 + 256 + units * (2 + 16) * G * (128 + 2) * 4)
    none = _dims(k=0, W=64)
    assert L.cmc_decode_attn_workspace_size(ctypes.byref(none)) == (
        256 + 256 + units * (0 + 1) * G * (128 + 2) * 4)
    many = _dims(B=40, Hkv=1, Hq=1, L=1, k=0, W=64)
    assert L.cmc_decode_attn_workspace_size(ctypes.byref(many)) == (
        256 + 512 + 40 * 1 * 1 * (4 + 128) * 4)
    assert L.cmc_decode_attn_workspace_size(ctypes.byref(_dims(d=80))) == 0


@host_only
def test_read_status_checks(L):
    flags = ctypes.c_uint32(0)
    assert L.cmc_read_status(0, 0, ctypes.byref(flags), None) == NULL


def test_binding_rejects_cpu_tensors():
    import torch
    with pytest.raises(ValueError, match="CUDA"):
        cmc.score_select(torch.zeros(1, 8), torch.zeros(1, 4, 8), 2)


@host_only
def test_tier1_gather_argument_checks(L):
    d = _dims()
    def g(bank=FAKE, idx=FAKE, out=FAKE, status=0, dims=d):
        return L.cmc_tier1_gather(bank, FAKE, idx, ctypes.byref(dims), out, FAKE, status, None)
    assert g(bank=0) == NULL
    assert g(idx=0) == NULL
    assert g(out=0) == NULL
    assert g(bank=FAKE + 8) == ALIGN
    assert g(idx=FAKE + 2) == ALIGN
    assert g(status=FAKE + 2) == ALIGN
    assert g(dims=_dims(k=101)) == RANGE
    assert g(dims=_dims(d=32)) == SHAPE
    assert g(dims=_dims(Hq=3)) not in (SHAPE,)  # query heads are ignored
    assert g(bank=0, idx=0, out=0, dims=_dims(k=0)) == 0  # k = 0: nothing to do
    assert L.cmc_tier1_gather(FAKE, FAKE, FAKE, None, FAKE, FAKE, 0, None) == NULL


def test_decode_attn_plan_argument_checks(L):
    ctas, launches = ctypes.c_int(0), ctypes.c_int(0)
    assert L.cmc_decode_attn_plan(None, 1, ctypes.byref(ctas), ctypes.byref(launches)) == NULL
    assert L.cmc_decode_attn_plan(ctypes.byref(_dims()), 1, None, ctypes.byref(launches)) == NULL
    assert L.cmc_decode_attn_plan(ctypes.byref(_dims(d=96)), 1, ctypes.byref(ctas),
                                  ctypes.byref(launches)) == SHAPE
    assert L.cmc_decode_attn_plan(ctypes.byref(_dims(k=101)), 0, ctypes.byref(ctas),
                                  ctypes.byref(launches)) == RANGE


@host_only
def test_decode_step_rope_argument_checks(L):
    d = _dims()
    def r(theta=10000.0, off=0, k_new=FAKE, dims=d, wsb=1 << 30):
        return L.cmc_decode_step_rope(FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, k_new, FAKE,
                                      ctypes.byref(dims), 0.0, theta, off, FAKE, FAKE, wsb, None)
    assert r(theta=0.0) == RANGE
    assert r(theta=-5.0) == RANGE
    assert r(theta=float("inf")) == RANGE
    assert r(theta=float("nan")) == RANGE
    assert r(off=-1) == RANGE
    assert r(k_new=0) == NULL
    assert r(dims=_dims(d=96)) == SHAPE
    assert r(wsb=16) == WORKSPACE


def test_question_select_workspace_size(L):
    # scores and squared norms (1,200 bytes each -> 1,280), 3 counters, 3
    # histograms of 2,048 counts, 3 argmax slots
    assert L.cmc_question_select_workspace_size(3, 100) == 2 * 1280 + 256 + 3 * 8192 + 256
    assert L.cmc_question_select_workspace_size(0, 100) == 0


@host_only
def test_question_select_argument_checks(L):
    def q(tok=FAKE, qlen=0, Lq=8, bank=FAKE, B=2, N=64, D=16, k=8, offs=FAKE, clen=FAKE, W=32,
          qv=FAKE, idx=FAKE, alpha=FAKE, start=FAKE, ws=FAKE, wsb=1 << 20):
        return L.cmc_question_select(tok, qlen, Lq, bank, B, N, D, k, offs, clen, W, qv, idx,
                                     alpha, start, ws, wsb, None)
    assert q(Lq=0) == SHAPE
    assert q(D=18) == SHAPE
    assert q(k=65) == RANGE
    assert q(W=0) == RANGE                       # localising needs a window
    assert q(tok=0) == NULL
    assert q(qv=0) == NULL
    assert q(idx=0) == NULL
    assert q(offs=0) == NULL                     # alpha/start requested without offsets
    assert q(ws=0) == NULL
    assert q(tok=FAKE + 4) == ALIGN
    assert q(alpha=FAKE + 2) == ALIGN
    assert q(wsb=100) == WORKSPACE
    # no localisation asked: offsets, lengths and W are not needed
    assert q(offs=0, clen=0, W=0, alpha=0, start=0) not in (NULL, RANGE, SHAPE, ALIGN, WORKSPACE)


@host_only
def test_bridge_epilogue_argument_checks(L):
    def b(x=FAKE, g=0, be=0, rows=4, D=64, eps=1e-5, nu=1.0, out=FAKE):
        return L.cmc_bridge_epilogue(x, g, be, rows, D, eps, nu, out, None)
    assert b(rows=0) == SHAPE
    assert b(D=66) == SHAPE
    assert b(D=16388) == SHAPE
    assert b(eps=0.0) == RANGE
    assert b(nu=-1.0) == RANGE
    assert b(nu=float("inf")) == RANGE
    assert b(x=0) == NULL
    assert b(out=0) == NULL
    assert b(x=FAKE + 4) == ALIGN
    assert b(g=FAKE + 8) == ALIGN


def test_denoise_workspace_size(L):
    # flags 2,000 -> 2,048; words 2 x 32 -> 256; counters 2 x 4 -> 256
    assert L.cmc_denoise_workspace_size(2, 1000) == 2048 + 256 + 256
    assert L.cmc_denoise_workspace_size(0, 10) == 0


@host_only
def test_denoise_argument_checks(L):
    def d(emb=FAKE, nt=0, B=2, n=100, H=64, g=3, tau=0.05, every=16, idx=FAKE, cnt=FAKE,
          ws=FAKE, wsb=1 << 20):
        return L.cmc_denoise(emb, nt, B, n, H, g, tau, every, idx, cnt, ws, wsb, None)
    assert d(H=66) == SHAPE
    assert d(n=0) == SHAPE
    assert d(g=0) == RANGE
    assert d(g=9) == RANGE
    assert d(every=-1) == RANGE
    assert d(tau=float("nan")) == RANGE
    assert d(emb=0) == NULL
    assert d(idx=0) == NULL
    assert d(emb=FAKE + 4) == ALIGN
    assert d(cnt=FAKE + 2) == ALIGN
    assert d(wsb=100) == WORKSPACE


@host_only
def test_stage_copies_argument_checks(L):
    def call(copies, n, wait_first=0):
        arr = (_lib.CmcCopy * max(1, len(copies)))()
        for i, (s, d, b) in enumerate(copies):
            arr[i].src, arr[i].dst, arr[i].bytes = s, d, b
        return L.cmc_stage_copies(ctypes.cast(arr, ctypes.c_void_p), n, wait_first, None)
    assert call([(FAKE, FAKE, 64)] * 4, 5) == RANGE
    assert call([(FAKE, FAKE, 64)], -1) == RANGE
    assert L.cmc_stage_copies(None, 1, 0, None) == NULL
    assert call([(0, FAKE, 64)], 1) == NULL
    assert call([(FAKE, 0, 64)], 1) == NULL
    assert call([(FAKE + 8, FAKE, 64)], 1) == ALIGN
    assert call([(FAKE, FAKE + 4, 64)], 1) == ALIGN
    assert call([(FAKE, FAKE, 40)], 1) == ALIGN


def test_l2_prefetch_setting_range(L):
    """The attention launches' prefetch depth: 0 to 64 tiles, else
    CMC_ERR_RANGE (host logic only; the default is put back)."""
    assert L.cmc_set_l2_prefetch_tiles(-1) == 3
    assert L.cmc_set_l2_prefetch_tiles(65) == 3
    assert L.cmc_set_l2_prefetch_tiles(0) == 0
    assert L.cmc_set_l2_prefetch_tiles(64) == 0
    assert L.cmc_set_l2_prefetch_tiles(5) == 0


def test_binding_sets_l2_prefetch():
    """The package-level binding of the prefetch setting (host logic only)."""
    cmc.set_l2_prefetch_tiles(0)
    cmc.set_l2_prefetch_tiles(5)
    with pytest.raises(cmc.CmcError):
        cmc.set_l2_prefetch_tiles(65)
