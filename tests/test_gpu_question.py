"""The question-side prologue on the GPU against the fp64 oracle: the pooled
question vector (within fp32 rounding), the Tier-1 selection (bit-exact, the
planted set), and the CME-guided window start (exact: the argmax of the CME
norms is taken on inputs whose top two squared norms differ by far more than
fp32 accumulation error, checked in each test)."""

import numpy as np
import pytest
import torch

import oracle
import paper_2609_25537_gb300 as cmc
from workloads import WORKLOADS, question_inputs, selection_inputs

pytestmark = pytest.mark.gpu


def _dev(a, dev):
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev)


def _norm_gap_ok(bank):
    for b in range(bank.shape[0]):
        sq = np.sort(np.einsum("ij,ij->i", bank[b].astype(np.float64), bank[b].astype(np.float64)))
        assert (sq[-1] - sq[-2]) / sq[-1] > 1e-5, "inputs too close to a norm tie for this test"


def _check(tokens, q_len, bank, k, offs, clen, W, dev, planted=None):
    q, idx, alpha, start = cmc.question_select(
        _dev(tokens, dev), _dev(bank, dev), k, q_len=None if q_len is None else _dev(q_len, dev),
        chunk_offset=_dev(offs, dev), ctx_len=_dev(clen, dev), W=W)
    ql = np.full(tokens.shape[0], tokens.shape[1], dtype=np.int32) if q_len is None else q_len
    rq, ridx, _, ralpha, rstart = oracle.question_select(tokens, ql, bank, k, offs, clen, W)
    torch.cuda.synchronize()
    np.testing.assert_allclose(q.cpu().numpy(), rq, rtol=1e-6, atol=1e-7)
    np.testing.assert_array_equal(idx.cpu().numpy(), ridx)
    if planted is not None:
        np.testing.assert_array_equal(idx.cpu().numpy(), planted)
    np.testing.assert_array_equal(alpha.cpu().numpy(), ralpha)
    np.testing.assert_array_equal(start.cpu().numpy(), rstart)


@pytest.mark.parametrize("name,batch,ratio", [
    ("tiny", None, 4), ("llama3_8b", None, 4), ("mistral_batched", range(0, 8), 4),
    ("long_context", range(0, 2), 8),
])
def test_question_prologue_workloads(cuda_device, name, batch, ratio):
    w = WORKLOADS[name]
    si = selection_inputs(w, batch=batch)
    qi = question_inputs(w, si, ratio=ratio, batch=batch)
    _norm_gap_ok(si.cme_bank)
    _check(qi.tokens, qi.q_len, si.cme_bank, w.k, qi.chunk_offset, qi.ctx_len, w.W, cuda_device,
           planted=si.planted_idx)


def test_question_prologue_edge_cases(cuda_device):
    """An empty question (zero vector: every score 0, so the first k CMEs),
    CMEs tied for the largest norm (lower index), a context shorter than the
    window (start 0), a window pushed against the context end, and k = 0."""
    rng = np.random.default_rng(11)
    B, Lq, N, D, W = 4, 6, 50, 32, 16
    tokens = rng.standard_normal((B, Lq, D)).astype(np.float32)
    bank = rng.standard_normal((B, N, D)).astype(np.float32)
    bank[1, 30] = bank[1, 7] = bank[1].max() * 3.0     # tied largest norms: 7 wins
    bank[3, 49] *= 4.0                                   # last chunk -> window at the end
    q_len = np.array([0, 6, 3, 1], dtype=np.int32)
    offs = np.tile((np.arange(N, dtype=np.int32) // 5) * 40, (B, 1))
    offs[3, 45:] = 395                                   # last chunk ends the context
    clen = np.array([400, 400, 10, 400], dtype=np.int32)
    for k in (5, 0):
        _check(tokens, q_len, bank, k, offs, clen, W, cuda_device)
    q, idx, alpha, start = cmc.question_select(_dev(tokens, cuda_device), _dev(bank, cuda_device),
                                               5, q_len=_dev(q_len, cuda_device),
                                               chunk_offset=_dev(offs, cuda_device),
                                               ctx_len=_dev(clen, cuda_device), W=W)
    assert idx[0].tolist() == [0, 1, 2, 3, 4]
    assert int(alpha[1]) == offs[1, 7]
    assert int(start[2]) == 0 and int(start[3]) == 400 - W
    # no q_len: every question uses all Lq rows
    _check(tokens, None, bank, 5, offs, clen, W, cuda_device)


def test_question_prologue_ties_inside_a_cta_and_workspace_reuse(cuda_device):
    """Largest norms tied inside one CTA's rows and across CTAs (the lowest
    index wins), in the one-launch path; the same workspace serves repeated
    calls and its completion counters, histograms and argmax slots are zero
    after each."""
    rng = np.random.default_rng(12)
    B, Lq, N, D, W, k = 3, 5, 64, 48, 16, 9
    tokens = rng.standard_normal((B, Lq, D)).astype(np.float32)
    bank = rng.standard_normal((B, N, D)).astype(np.float32)
    big = np.abs(bank).max() * 4.0
    bank[0, 13] = bank[0, 12] = big       # the same CTA for every rows-per-CTA up to 8: 12 wins
    bank[1, 40] = bank[1, 3] = big        # different CTAs: 3 wins
    bank[2, 63] = big                     # the last row
    q_len = np.array([5, 2, 4], dtype=np.int32)
    offs = np.tile(np.arange(N, dtype=np.int32) * 7, (B, 1))
    clen = np.full(B, 7 * N, dtype=np.int32)
    ws = torch.zeros(cmc.lib().cmc_question_select_workspace_size(B, N), dtype=torch.uint8,
                     device=cuda_device)
    rq, ridx, _, ralpha, rstart = oracle.question_select(tokens, q_len, bank, k, offs, clen, W)
    assert ralpha.tolist() == [offs[0, 12], offs[1, 3], offs[2, 63]]
    for _ in range(3):
        q, idx, alpha, start = cmc.question_select(
            _dev(tokens, cuda_device), _dev(bank, cuda_device), k,
            q_len=_dev(q_len, cuda_device), chunk_offset=_dev(offs, cuda_device),
            ctx_len=_dev(clen, cuda_device), W=W, workspace=ws)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(idx.cpu().numpy(), ridx)
        np.testing.assert_array_equal(alpha.cpu().numpy(), ralpha)
        np.testing.assert_array_equal(start.cpu().numpy(), rstart)
        tail = ws[2 * (-(-B * N * 4 // 256) * 256):].cpu().numpy()
        assert not tail.any(), "counters, histograms or argmax slots not left at zero"
