"""The allocation-free selection entry point, cmc_score_select_static.

It exists for callers that cannot give the library a workspace (an engine
that has reserved all free HBM for its KV-cache pool and allows no later
allocation, or a C host program with no device allocator of its own).  These
tests call it through the C ABI and check that it selects exactly what the
workspace-based cmc_score_select selects (the index set is compared
bit-exactly, as everywhere else), on two calls in a row that reuse the shared
device scratch array.  This file is named to be collected last.
"""

import ctypes

import numpy as np
import pytest
import torch

import paper_2609_25537_gb300 as cmc
from paper_2609_25537_gb300 import _lib
from workloads import WORKLOADS, selection_inputs

pytestmark = pytest.mark.gpu

SHAPE = 2


def _static_select(question_emb, cme_bank, k):
    B, N, D = cme_bank.shape
    idx = torch.full((B, k), -7, dtype=torch.int32, device=cme_bank.device)
    st = cmc.lib().cmc_score_select_static(
        ctypes.c_void_p(question_emb.data_ptr()), ctypes.c_void_p(cme_bank.data_ptr()),
        B, N, D, k, ctypes.c_void_p(idx.data_ptr()),
        ctypes.c_void_p(torch.cuda.current_stream(cme_bank.device).cuda_stream))
    assert st == 0, _lib.STATUS.get(st, st)
    return idx


def test_static_select_matches_workspace_select_on_two_calls(cuda_device):
    calls = [(WORKLOADS["llama3_8b"], None), (WORKLOADS["mistral_batched"], range(0, 16))]
    for w, batch in calls:
        si = selection_inputs(w, batch=batch)
        q = torch.from_numpy(si.question_emb).to(cuda_device)
        bank = torch.from_numpy(si.cme_bank).to(cuda_device)
        got = _static_select(q, bank, w.k)
        want = cmc.score_select(q, bank, w.k)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(got.cpu().numpy(), want.cpu().numpy())
        np.testing.assert_array_equal(got.cpu().numpy(), si.planted_idx)


def test_static_select_rejects_sizes_beyond_its_array(cuda_device):
    B, N, D = 2, _lib.STATIC_SCORES_MAX // 2 + 1, 4
    q = torch.ones((B, D), dtype=torch.float32, device=cuda_device)
    bank = torch.ones((1, 1, D), dtype=torch.float32, device=cuda_device)  # never read
    idx = torch.empty((B, 4), dtype=torch.int32, device=cuda_device)
    st = cmc.lib().cmc_score_select_static(
        ctypes.c_void_p(q.data_ptr()), ctypes.c_void_p(bank.data_ptr()), B, N, D, 4,
        ctypes.c_void_p(idx.data_ptr()), None)
    assert st == SHAPE
