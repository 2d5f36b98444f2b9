"""Tier-1 scoring and selection on the GPU against the fp64 oracle.

The selected index set is compared bit-exactly (as an ordered array); scores
within 1e-5 absolute (fp32 accumulation over D <= 4096 terms of a cosine).

Both launch paths run on every case: one launch (a workspace given, N <= 8192,
D <= 4096: the CTA that completes a sequence's scores selects it) and two
launches (no workspace, scores_out given, reached through the C ABI; also the
path of larger banks).  They must select the same rows."""

import ctypes

import numpy as np
import pytest
import torch

import oracle
import paper_2609_25537_gb300 as cmc
from workloads import WORKLOADS, selection_inputs
from workloads.configs import ablation_workload
from _gpu_helpers import dev_f32

pytestmark = pytest.mark.gpu

SCORE_ATOL = 1e-5


def _two_launch(qd, bd, k):
    """cmc_score_select without a workspace (scores_out given): the scoring
    kernel, then the selection kernel."""
    B, N, D = bd.shape
    idx = torch.full((B, k), -1, dtype=torch.int32, device=bd.device)
    sc = torch.empty((B, N), dtype=torch.float32, device=bd.device)
    st = cmc.lib().cmc_score_select(
        ctypes.c_void_p(qd.data_ptr()), ctypes.c_void_p(bd.data_ptr()), B, N, D, k,
        ctypes.c_void_p(idx.data_ptr()), ctypes.c_void_p(sc.data_ptr()), None, 0,
        ctypes.c_void_p(torch.cuda.current_stream(bd.device).cuda_stream))
    assert st == 0
    return idx, sc


def _run(q, bank, k, dev):
    qd, bd = dev_f32(q, dev), dev_f32(bank, dev)
    scores = torch.empty(bank.shape[:2], dtype=torch.float32, device=dev)
    idx = cmc.score_select(qd, bd, k, scores_out=scores)
    # the workspace path (no scores_out) must select the same rows
    idx2 = cmc.score_select(qd, bd, k)
    # and so must the two-launch path
    idx3, scores3 = _two_launch(qd, bd, k)
    torch.cuda.synchronize()
    assert torch.equal(idx, idx2)
    assert torch.equal(idx, idx3)
    assert (scores - scores3).abs().max().item() <= 2 * SCORE_ATOL
    return idx.cpu().numpy(), scores.cpu().numpy()


@pytest.mark.parametrize("name,batch", [
    ("tiny", None), ("llama3_8b", None), ("mistral_batched", None),
    ("long_context", range(0, 2)),
])
def test_select_workloads(cuda_device, name, batch):
    w = WORKLOADS[name]
    si = selection_inputs(w, batch=batch)
    idx, scores = _run(si.question_emb, si.cme_bank, w.k, cuda_device)
    ref_idx, ref_scores = oracle.score_select(si.question_emb, si.cme_bank, w.k)
    np.testing.assert_array_equal(idx, ref_idx)
    np.testing.assert_array_equal(idx, si.planted_idx)
    assert np.abs(scores - ref_scores).max() <= SCORE_ATOL


@pytest.mark.parametrize("k", [0, 64, 256, 1024])
def test_select_ablation_k(cuda_device, k):
    w = ablation_workload(k, 512, 16)
    si = selection_inputs(w)
    idx, _ = _run(si.question_emb, si.cme_bank, w.k, cuda_device)
    ref_idx, _ = oracle.score_select(si.question_emb, si.cme_bank, w.k)
    np.testing.assert_array_equal(idx, ref_idx)


def test_select_ties_go_to_lower_index(cuda_device):
    rng = np.random.default_rng(7)
    B, N, D = 3, 700, 64
    q = rng.standard_normal((B, D)).astype(np.float32)
    bank = rng.standard_normal((B, N, D)).astype(np.float32)
    # three bit-identical rows at the top; k = 2 must keep the two lowest indices
    for b in range(B):
        top = (q[b] * 3.0 + 0.01 * rng.standard_normal(D)).astype(np.float32)
        for j in (5, 300, 650):
            bank[b, j] = top
    idx, scores = _run(q, bank, 2, cuda_device)
    assert idx.tolist() == [[5, 300]] * B
    assert np.all(scores[:, 5] == scores[:, 300]) and np.all(scores[:, 300] == scores[:, 650])
    # duplicates straddling the cut deep in the ranking
    k = 100
    ref_scores = oracle.cosine_scores(q, bank)
    for b in range(B):
        order = np.argsort(-ref_scores[b], kind="stable")
        cut_row = bank[b, order[k - 1]].copy()
        for j in (order[k - 1], order[k + 5], 699):
            bank[b, j] = cut_row
    idx, _ = _run(q, bank, k, cuda_device)
    ref_idx, _ = oracle.score_select(q, bank, k)
    np.testing.assert_array_equal(idx, ref_idx)


# the last three: a cluster of 8 selection CTAs per sequence (N > 8,192),
# keys split across their shared memories (also unevenly: 50,001 = 8 x 6,250
# + 1), and one CTA re-reading the keys from global memory (N / 8 > 49,152)
#
# One launch for small banks (CTAs of R <= 8 rows of one sequence, R dividing
# N, one wave of one CTA per SM; D <= 4096): R = 8 (1000, 1024, 1216 = 8 x
# 152 rows), R = 7 (777), R = 3 (B = 7, N = 33), R = 1 (prime N = 37, B = 4),
# R = 5 (N = 5), and the two-key-per-thread selection (N = 1216); D from 4 to
# 4096, one float4 per thread or fewer.  Two launches otherwise (D = 4100, and
# the larger banks).
@pytest.mark.parametrize("N,D,k,B", [
    (1, 4, 1, 3), (1, 4, 0, 3), (5, 8, 5, 3), (1000, 36, 999, 3), (1025, 512, 17, 3),
    (3000, 4, 1500, 3), (4096, 128, 4095, 3), (9000, 8, 1234, 3), (50001, 4, 777, 3),
    (400003, 4, 1000, 3), (8192, 16, 4000, 2), (8193, 16, 100, 2), (1000, 36, 999, 1),
    (1024, 4096, 1023, 1), (1024, 2048, 1, 1), (1216, 64, 300, 1), (777, 4, 50, 1),
    (33, 4096, 5, 7), (37, 100, 9, 4), (300, 4100, 50, 2), (1024, 256, 100, 40)])
def test_select_edge_shapes(cuda_device, N, D, k, B):
    """Random banks (no planted margin), through both launch paths."""
    rng = np.random.default_rng(N + D + k)
    q = rng.standard_normal((B, D)).astype(np.float32)
    bank = rng.standard_normal((B, N, D)).astype(np.float32)
    idx, scores = _run(q, bank, k, cuda_device)
    ref_idx, ref_scores = oracle.score_select(q, bank, k)
    assert np.abs(scores - ref_scores).max() <= SCORE_ATOL
    # without a planted margin, compare where the float32 decision is unambiguous
    for b in range(B):
        s = np.sort(ref_scores[b])[::-1]
        if k in (0, N) or s[k - 1] - s[k] > 1e-5:
            np.testing.assert_array_equal(idx[b], ref_idx[b])
        assert idx[b].tolist() == sorted(set(idx[b].tolist()))
        assert len(idx[b]) == k


def test_select_zero_vectors(cuda_device):
    B, N, D = 2, 40, 16
    rng = np.random.default_rng(3)
    q = rng.standard_normal((B, D)).astype(np.float32)
    q[1] = 0.0                                    # zero question: every score 0
    bank = rng.standard_normal((B, N, D)).astype(np.float32)
    bank[0, 7] = 0.0                              # zero CME: score 0
    idx, scores = _run(q, bank, 10, cuda_device)
    assert scores[0, 7] == 0.0 and np.all(scores[1] == 0.0)
    assert idx[1].tolist() == list(range(10))
    ref_idx, _ = oracle.score_select(q, bank, 10)
    np.testing.assert_array_equal(idx, ref_idx)


def test_select_negative_and_signed_zero_scores(cuda_device):
    # orthogonal rows give +-0 dot products; -0 and +0 must tie (lower index wins)
    B, N, D = 1, 8, 4
    q = np.array([[1.0, 0.0, 0.0, 0.0]], dtype=np.float32)
    bank = np.zeros((B, N, D), dtype=np.float32)
    bank[0, :, 1] = 1.0
    bank[0, 0] = [-1.0, 0.0, 0.0, 0.0]   # score -1
    bank[0, 3] = [-0.0, 2.0, 0.0, 0.0]   # dot -0
    bank[0, 6] = [0.5, 0.5, 0.0, 0.0]    # positive
    idx, scores = _run(q, bank, 3, cuda_device)
    assert idx[0].tolist() == [1, 2, 6]
    assert not np.signbit(scores[0, 3])


def _bank_of_scores(s):
    """Rows whose cosine with q = e_0 is s_j: m_j = (s_j, sqrt(1 - s_j^2), 0, ...)."""
    N, D = len(s), 64
    bank = np.zeros((1, N, D), dtype=np.float32)
    bank[0, :, 0] = s
    bank[0, :, 1] = np.sqrt(1.0 - np.asarray(s, dtype=np.float64) ** 2)
    q = np.zeros((1, D), dtype=np.float32)
    q[0, 0] = 1.0
    return q, bank


@pytest.mark.parametrize("case", ["level1_single", "level1_whole_bin", "level2", "level3_ties"])
def test_select_search_levels(cuda_device, case):
    """The one-launch selection's histogram search ends at the first level
    whose chosen bin holds exactly the keys still to take; banks built so
    that it ends at each level (top 11 key bits: the k-th score alone in
    [0.5, 0.625), or that bin taken whole; top 21 bits: 0.56 among many
    0.52; all 32: 0.56 three times, two of them taken, lowest indices
    first).  N = 1,024, k = 100, against the oracle and the two-launch
    path."""
    N, k = 1024, 100
    rng = np.random.default_rng(11)
    s = np.full(N, 0.1)
    s[rng.choice(N, 300, replace=False)] = 0.3
    perm = rng.permutation(N)
    if case == "level1_single":
        s[perm[:k - 1]] = 0.9
        s[perm[k - 1]] = 0.55
    elif case == "level1_whole_bin":
        s[perm[:k - 3]] = 0.9
        s[perm[k - 3:k]] = 0.55
    elif case == "level2":
        s[perm[:k - 1]] = 0.9
        s[perm[k - 1]] = 0.56
        s[perm[k:k + 200]] = 0.52
    else:
        s[perm[:k - 2]] = 0.9
        s[perm[k - 2:k + 1]] = 0.56
        s[perm[k + 1:k + 200]] = 0.52
    q, bank = _bank_of_scores(s)
    idx, _ = _run(q, bank, k, cuda_device)
    ref_idx, _ = oracle.score_select(q, bank, k)
    np.testing.assert_array_equal(idx, ref_idx)
    if case == "level3_ties":
        tied = np.sort(perm[k - 2:k + 1])
        assert set(tied[:2]) <= set(idx[0].tolist()) and tied[2] not in idx[0]


@pytest.mark.parametrize("name,B", [("mistral_batched", 8), ("llama3_8b", 1), ("tiny", 2)])
def test_one_launch_counters_reset_across_calls(cuda_device, name, B):
    """One workspace over calls on different banks (the one-launch path at the
    Llama and tiny shapes, two launches for the Mistral batch): every call
    selects exactly the planted set, and leaves the completion counters and
    the score histograms at zero."""
    w = WORKLOADS[name]
    ws = torch.zeros(cmc.score_select_workspace_size(B, w.N), dtype=torch.uint8,
                     device=cuda_device)
    scores_bytes = -(-B * w.N * 4 // 256) * 256
    for batch in (range(0, B), range(B, 2 * B), range(0, B)):
        si = selection_inputs(w, batch=batch)
        idx = cmc.score_select(dev_f32(si.question_emb, cuda_device),
                               dev_f32(si.cme_bank, cuda_device), w.k, workspace=ws)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(idx.cpu().numpy(), si.planted_idx)
        assert not ws[scores_bytes:].cpu().numpy().any(), "counters or histograms left non-zero"
