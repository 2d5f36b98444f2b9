"""The seeded generator: determinism, bf16 rounding and the planted margin."""

import numpy as np
import pytest
import torch

import oracle
from workloads import (WORKLOADS, selection_inputs, kv_inputs, step_inputs,
                       f32_to_bf16_bits, bf16_bits_to_f32)
from workloads.configs import ablation_workloads, full_window_workload


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = np.concatenate([
        rng.standard_normal(100000).astype(np.float32) * 3,
        # exact halfway cases: ties go to even
        np.array([1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -(1.0 + 2 ** -8), 0.0, -0.0],
                 dtype=np.float32),
    ])
    ours = f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(ours, ref)
    back = bf16_bits_to_f32(ours)
    np.testing.assert_array_equal(back, torch.from_numpy(ref.view(np.int16)).view(
        torch.bfloat16).float().numpy())


def test_generation_is_deterministic_and_per_sequence():
    w = WORKLOADS["tiny"].with_(B=3)
    a = kv_inputs(w)
    b = kv_inputs(w, batch=range(1, 2))
    np.testing.assert_array_equal(a.tier1_k[1:2], b.tier1_k)
    np.testing.assert_array_equal(a.ring_v[1:2], b.ring_v)
    s1 = selection_inputs(w)
    s2 = selection_inputs(w)
    np.testing.assert_array_equal(s1.cme_bank, s2.cme_bank)
    np.testing.assert_array_equal(s1.planted_idx, s2.planted_idx)
    t1 = step_inputs(w, 5)
    t2 = step_inputs(w, 5)
    np.testing.assert_array_equal(t1.q, t2.q)
    assert not np.array_equal(step_inputs(w, 6).q, t1.q)


def test_distributions():
    w = WORKLOADS["llama3_8b"]
    kv = kv_inputs(w.with_(L=2))
    x = bf16_bits_to_f32(kv.tier1_k)
    assert abs(x.std() - w.kv_std) < 0.01 * w.kv_std
    assert abs(x.mean()) < 0.01 * w.kv_std
    assert np.all(kv.pos0 == w.W)
    si = selection_inputs(w)
    assert abs(si.cme_bank.std() - w.emb_std) < 0.02 * w.emb_std
    norms = np.linalg.norm(si.cme_bank[0], axis=1)
    assert abs(norms.mean() - 1.0) < 0.02


def test_partial_fill_leaves_unused_slots_zero():
    w = WORKLOADS["tiny"].with_(B=2, W0=(5, 128))
    kv = kv_inputs(w)
    assert kv.pos0.tolist() == [5, 128]
    assert np.all(kv.ring_k[0, :, :, 5:] == 0)
    assert np.any(kv.ring_k[0, :, :, :5] != 0)


@pytest.mark.parametrize("name", ["mistral_batched", "long_context"])
def test_planted_gap_large_banks(name):
    """One sequence of each large bank: the oracle's fp64 gap at the top-k cut
    is above 1e-4 and its selection is the planted set."""
    w = WORKLOADS[name]
    si = selection_inputs(w, batch=range(0, 1))
    idx, scores = oracle.score_select(si.question_emb, si.cme_bank, w.k)
    np.testing.assert_array_equal(idx, si.planted_idx)
    srt = np.sort(scores[0])[::-1]
    assert srt[w.k - 1] - srt[w.k] >= 1e-4


def test_ablation_grid_shape():
    ws = ablation_workloads()
    assert len(ws) == 45
    assert {w.k for w in ws} == {0, 64, 256, 1024}
    fw = full_window_workload(T=8)
    assert fw.W >= fw.fill()[0] + fw.T and fw.k == fw.N
