"""Pins of the fp64 oracle against facts fixed outside it.

Each test checks the oracle against something other than its own formula:
closed forms, brute force over all candidate answers, library routines
(scipy / torch fp64) on the special cases they cover, and invariants of the
method (Section 2.5: cosine scoring, top-K with document-order re-ordering,
the bounded two-tier cache).  A plausible slip in the oracle (a dropped norm,
a wrong sign, a transposed operand, an off-by-one in the ring, the wrong GQA
head mapping, a missing scale) fails at least one of them.
"""

import itertools
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from workloads import (WORKLOADS, selection_inputs, kv_inputs, step_inputs,
                       f32_to_bf16_bits, bf16_bits_to_f32)
from workloads.configs import Workload

pytestmark = pytest.mark.filterwarnings("ignore::DeprecationWarning")


# ----------------------------------------------------------------------------
# Cosine scoring (Section 2.5, score_j)
# ----------------------------------------------------------------------------

def test_cosine_closed_forms():
    q = np.array([[3.0, 4.0]])
    bank = np.array([[[4.0, 3.0],     # 24 / 25
                      [6.0, 8.0],     # parallel: 1
                      [-3.0, -4.0],   # antiparallel: -1
                      [-4.0, 3.0],    # orthogonal: 0
                      [0.0, 0.0],     # zero vector: 0 (reading)
                      [0.0, 5.0]]])   # 20 / 25
    s = oracle.cosine_scores(q, bank)
    assert s.shape == (1, 6)
    np.testing.assert_allclose(s[0], [24 / 25, 1.0, -1.0, 0.0, 0.0, 0.8], rtol=0, atol=1e-15)


def test_cosine_zero_question_gives_zero_scores():
    s = oracle.cosine_scores(np.zeros((1, 8)), np.ones((1, 5, 8)))
    assert np.all(s == 0.0)


def test_cosine_against_scipy_and_torch():
    rng = np.random.default_rng(11)
    q = rng.standard_normal((3, 37))
    bank = rng.standard_normal((3, 50, 37)) * rng.uniform(0.1, 10, size=(3, 50, 1))
    s = oracle.cosine_scores(q, bank)
    t = F.cosine_similarity(torch.from_numpy(bank), torch.from_numpy(q)[:, None, :], dim=-1)
    np.testing.assert_allclose(s, t.numpy(), rtol=0, atol=1e-13)
    spatial = pytest.importorskip("scipy.spatial.distance")
    for b in range(3):
        for j in range(0, 50, 7):
            assert abs(s[b, j] - (1.0 - spatial.cosine(bank[b, j], q[b]))) < 1e-13


def test_cosine_scale_invariance_and_sign():
    rng = np.random.default_rng(12)
    q = rng.standard_normal((1, 64))
    bank = rng.standard_normal((1, 20, 64))
    c = rng.uniform(0.01, 100.0, size=(1, 20, 1))
    s = oracle.cosine_scores(q, bank)
    np.testing.assert_allclose(oracle.cosine_scores(q, bank * c), s, rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(oracle.cosine_scores(q * 7.5, bank), s, rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(oracle.cosine_scores(q, -bank), -s, rtol=0, atol=0)
    assert np.all(np.abs(s) <= 1.0)


# ----------------------------------------------------------------------------
# Top-K selection, re-ordered by document position (Section 2.5)
# ----------------------------------------------------------------------------

def _brute_force_topk(s: np.ndarray, k: int):
    """The unique k-subset S such that every kept j beats every dropped i:
    s_j > s_i, or s_j == s_i and j < i (ties to the lower index)."""
    N = len(s)
    found = []
    for S in itertools.combinations(range(N), k):
        inside = set(S)
        ok = all((s[j] > s[i]) or (s[j] == s[i] and j < i)
                 for j in inside for i in range(N) if i not in inside)
        if ok:
            found.append(S)
    assert len(found) == 1
    return list(found[0])


@pytest.mark.parametrize("seed", range(6))
def test_select_brute_force(seed):
    rng = np.random.default_rng(seed)
    N = 7
    # few distinct values, so ties straddle the cut often
    s = rng.integers(-2, 3, size=(1, N)).astype(np.float64) / 4.0
    for k in range(N + 1):
        got = oracle.select_top_k(s, k)[0].tolist()
        assert got == _brute_force_topk(s[0].astype(np.float32), k)
        assert got == sorted(got)


def test_select_ties_go_to_lower_index():
    s = np.full((2, 10), 0.25)
    np.testing.assert_array_equal(oracle.select_top_k(s, 4), [[0, 1, 2, 3]] * 2)
    s = np.array([[0.1, 0.5, 0.3, 0.5, 0.5, 0.2]])
    np.testing.assert_array_equal(oracle.select_top_k(s, 2), [[1, 3]])
    np.testing.assert_array_equal(oracle.select_top_k(s, 4), [[1, 2, 3, 4]])


def test_select_decides_in_float32():
    # 0.5 and 0.5 + 1e-12 are the same float32: a tie, so the lower index wins.
    s = np.array([[0.5, 0.5 + 1e-12, 0.1]])
    np.testing.assert_array_equal(oracle.select_top_k(s, 1), [[0]])
    # 0.5 and 0.5 + 1e-6 differ in float32: the larger wins.
    s = np.array([[0.5, 0.5 + 1e-6, 0.1]])
    np.testing.assert_array_equal(oracle.select_top_k(s, 1), [[1]])


def test_select_edges():
    s = np.random.default_rng(3).standard_normal((2, 9))
    assert oracle.select_top_k(s, 0).shape == (2, 0)
    np.testing.assert_array_equal(oracle.select_top_k(s, 9), [list(range(9))] * 2)
    with pytest.raises(ValueError):
        oracle.select_top_k(s, 10)


def test_select_recovers_rows_parallel_to_question():
    # rows built as a positive multiple of q plus tiny noise outrank all others
    rng = np.random.default_rng(5)
    D, N, k = 64, 40, 6
    q = rng.standard_normal((1, D))
    bank = rng.standard_normal((1, N, D))
    chosen = [3, 9, 17, 18, 30, 39]
    for j in chosen:
        bank[0, j] = rng.uniform(0.5, 3.0) * q[0] + 1e-3 * rng.standard_normal(D)
    idx, _ = oracle.score_select(q, bank, k)
    assert idx[0].tolist() == chosen


@pytest.mark.parametrize("name", ["tiny", "llama3_8b"])
def test_selection_matches_planted_set(name):
    w = WORKLOADS[name]
    si = selection_inputs(w)
    idx, scores = oracle.score_select(si.question_emb, si.cme_bank, w.k)
    np.testing.assert_array_equal(idx, si.planted_idx)
    # the planted gap at the cut survives float32 rounding of the inputs
    for b in range(w.B):
        srt = np.sort(scores[b])[::-1]
        assert srt[w.k - 1] - srt[w.k] >= 1e-4


# ----------------------------------------------------------------------------
# Tier-2 ring (Section 2.5, bounded two-tier cache)
# ----------------------------------------------------------------------------

def test_ring_equals_last_w_tokens():
    rng = np.random.default_rng(21)
    B, L, H, W, d = 2, 2, 3, 5, 4
    fill = [2, 5]
    ring_k = np.zeros((B, L, H, W, d))
    ring_v = np.zeros((B, L, H, W, d))
    hist_k = [[] for _ in range(B)]
    hist_v = [[] for _ in range(B)]
    pos = np.zeros(B, dtype=np.int64)
    for b in range(B):
        for t in range(fill[b]):
            kt = rng.standard_normal((L, H, d))
            vt = rng.standard_normal((L, H, d))
            ring_k[b, :, :, t] = kt
            ring_v[b, :, :, t] = vt
            hist_k[b].append(kt)
            hist_v[b].append(vt)
        pos[b] = fill[b]
    for step in range(13):
        kn = rng.standard_normal((B, L, H, d))
        vn = rng.standard_normal((B, L, H, d))
        before = pos.copy()
        oracle.window_append(ring_k, ring_v, pos, kn, vn)
        np.testing.assert_array_equal(pos, before + 1)
        for b in range(B):
            hist_k[b].append(kn[b])
            hist_v[b].append(vn[b])
            slots = list(oracle.window_slots(pos[b], W))
            assert len(slots) == min(len(hist_k[b]), W)
            got = sorted(ring_k[b, 0, 0, s, 0] for s in slots)
            want = sorted(x[0, 0, 0] for x in hist_k[b][-W:])
            assert got == want
            # token number p sits in slot p mod W
            p = int(pos[b]) - 1
            np.testing.assert_array_equal(ring_k[b, :, :, p % W], kn[b])


# ----------------------------------------------------------------------------
# Decode attention over [Tier-1 | Tier-2]
# ----------------------------------------------------------------------------

def test_attention_closed_forms():
    d = 2
    v1 = np.array([1.0, -2.0])
    v2 = np.array([4.0, 8.0])
    # logits ln 3 and 0 -> weights 3/4 and 1/4
    q = np.array([1.0, 0.0])
    K = np.array([[math.log(3.0), 0.0], [0.0, 0.0]])
    out = oracle.softmax_attention(q, K, np.stack([v1, v2]), scale=1.0)
    np.testing.assert_allclose(out, 0.75 * v1 + 0.25 * v2, rtol=0, atol=1e-15)
    # one key: its value
    out = oracle.softmax_attention(q, K[:1], v1[None], scale=3.0)
    np.testing.assert_allclose(out, v1, rtol=0, atol=0)
    # zero query: the mean of the values
    rng = np.random.default_rng(2)
    V = rng.standard_normal((9, d))
    out = oracle.softmax_attention(np.zeros(d), rng.standard_normal((9, d)), V, scale=1.0)
    np.testing.assert_allclose(out, V.mean(0), rtol=0, atol=1e-15)
    # empty cache: zeros
    assert np.all(oracle.softmax_attention(q, np.zeros((0, d)), np.zeros((0, d)), 1.0) == 0)


def test_attention_is_stable_for_large_logits():
    q = np.array([1.0, 0.0])
    K = np.array([[2000.0, 0.0], [1000.0, 0.0], [-5.0, 0.0]])
    V = np.array([[1.0, 2.0], [3.0, 4.0], [5.0, 6.0]])
    out = oracle.softmax_attention(q, K, V, scale=1.0)
    np.testing.assert_allclose(out, V[0], rtol=0, atol=0)


def _small_problem(seed, B=2, L=2, Hq=6, Hkv=2, d=8, N=11, k=4, W=5, fill=(3, 5)):
    rng = np.random.default_rng(seed)
    t1k = rng.standard_normal((B, L, Hkv, N, d))
    t1v = rng.standard_normal((B, L, Hkv, N, d))
    q = rng.standard_normal((B, L, Hq, d))
    idx = np.stack([np.sort(rng.choice(N, size=k, replace=False)) for _ in range(B)])
    ring_k = np.zeros((B, L, Hkv, W, d))
    ring_v = np.zeros((B, L, Hkv, W, d))
    hist = []
    pos = np.zeros(B, dtype=np.int64)
    for b in range(B):
        hk = rng.standard_normal((fill[b], L, Hkv, d))
        hv = rng.standard_normal((fill[b], L, Hkv, d))
        ring_k[b, :, :, : fill[b]] = hk.transpose(1, 2, 0, 3)
        ring_v[b, :, :, : fill[b]] = hv.transpose(1, 2, 0, 3)
        hist.append(([*hk], [*hv]))
        pos[b] = fill[b]
    return dict(q=q, t1k=t1k, t1v=t1v, idx=idx, ring_k=ring_k, ring_v=ring_v, pos=pos,
                hist=hist, rng=rng)


def _sdpa(q, K, V, scale=None):
    """torch fp64 scaled_dot_product_attention of one query over K, V."""
    out = F.scaled_dot_product_attention(
        torch.from_numpy(q)[None, None, None, :], torch.from_numpy(K)[None, None],
        torch.from_numpy(V)[None, None], scale=scale)
    return out[0, 0, 0].numpy()


def test_two_tier_attention_against_sdpa_with_history():
    """Keys assembled independently (selected bank rows + the last W tokens of
    the linear token history, GQA head h -> h // (Hq/Hkv)) and attended by the
    library routine."""
    P = _small_problem(31)
    q, t1k, t1v, idx = P["q"], P["t1k"], P["t1v"], P["idx"]
    ring_k, ring_v, pos, hist, rng = P["ring_k"], P["ring_v"], P["pos"], P["hist"], P["rng"]
    B, L, Hq, d = q.shape
    Hkv, W = ring_k.shape[2], ring_k.shape[3]
    G = Hq // Hkv
    for step in range(9):   # crosses the wrap of both sequences
        kn = rng.standard_normal((B, L, Hkv, d))
        vn = rng.standard_normal((B, L, Hkv, d))
        qs = rng.standard_normal((B, L, Hq, d))
        out = oracle.decode_step(qs, t1k, t1v, idx, ring_k, ring_v, pos, kn, vn)
        for b in range(B):
            hist[b][0].append(kn[b])
            hist[b][1].append(vn[b])
            lastk = np.stack(hist[b][0][-W:])
            lastv = np.stack(hist[b][1][-W:])
            for l in range(L):
                kv_k = torch.from_numpy(t1k[b, l]).repeat_interleave(G, dim=0).numpy()
                kv_v = torch.from_numpy(t1v[b, l]).repeat_interleave(G, dim=0).numpy()
                wk = torch.from_numpy(lastk[:, l]).repeat_interleave(G, dim=1).numpy()
                wv = torch.from_numpy(lastv[:, l]).repeat_interleave(G, dim=1).numpy()
                for h in range(Hq):
                    K = np.concatenate([kv_k[h][idx[b]], wk[:, h]])
                    V = np.concatenate([kv_v[h][idx[b]], wv[:, h]])
                    np.testing.assert_allclose(out[b, l, h], _sdpa(qs[b, l, h], K, V),
                                               rtol=1e-12, atol=1e-12)


def test_all_cmes_and_unbounded_window_equal_plain_attention():
    """k = N and a window that never evicts: the two-tier cache holds every
    token, so the result is plain attention over [bank | all tokens]."""
    rng = np.random.default_rng(41)
    B, L, Hq, Hkv, d, N, W = 1, 1, 4, 2, 16, 9, 32
    t1k = rng.standard_normal((B, L, Hkv, N, d))
    t1v = rng.standard_normal((B, L, Hkv, N, d))
    ring_k = np.zeros((B, L, Hkv, W, d))
    ring_v = np.zeros((B, L, Hkv, W, d))
    pos = np.zeros(B, dtype=np.int64)
    toks_k, toks_v = [], []
    scores = rng.standard_normal((B, N))
    idx = oracle.select_top_k(scores, N)
    np.testing.assert_array_equal(idx[0], np.arange(N))
    for step in range(20):
        kn = rng.standard_normal((B, L, Hkv, d))
        vn = rng.standard_normal((B, L, Hkv, d))
        qs = rng.standard_normal((B, L, Hq, d)) * 2.0
        out = oracle.decode_step(qs, t1k, t1v, idx, ring_k, ring_v, pos, kn, vn)
        toks_k.append(kn[0, 0])
        toks_v.append(vn[0, 0])
        for h in range(Hq):
            g = h // (Hq // Hkv)
            K = np.concatenate([t1k[0, 0, g], np.stack(toks_k)[:, g]])
            V = np.concatenate([t1v[0, 0, g], np.stack(toks_v)[:, g]])
            np.testing.assert_allclose(out[0, 0, h], _sdpa(qs[0, 0, h], K, V),
                                       rtol=1e-12, atol=1e-12)


def test_k_zero_is_window_only_attention():
    P = _small_problem(51, k=0)
    q, ring_k, ring_v, pos = P["q"], P["ring_k"], P["ring_v"], P["pos"]
    out = oracle.two_tier_attention(q, P["t1k"], P["t1v"], None, ring_k, ring_v, pos)
    out2 = oracle.two_tier_attention(q, P["t1k"], P["t1v"], np.zeros((2, 0), np.int64),
                                     ring_k, ring_v, pos)
    np.testing.assert_array_equal(out, out2)
    B, L, Hq, d = q.shape
    G = Hq // ring_k.shape[2]
    for b in range(B):
        n = int(pos[b])
        for l in range(L):
            for h in range(Hq):
                K = ring_k[b, l, h // G, :n]
                V = ring_v[b, l, h // G, :n]
                np.testing.assert_allclose(out[b, l, h], _sdpa(q[b, l, h], K, V),
                                           rtol=1e-12, atol=1e-12)


def test_attention_key_order_and_scale():
    P = _small_problem(61)
    q, t1k, t1v, idx = P["q"], P["t1k"], P["t1v"], P["idx"]
    base = oracle.two_tier_attention(q, t1k, t1v, idx, P["ring_k"], P["ring_v"], P["pos"])
    # permuting the selected rows or the ring slots leaves the output unchanged
    rev = idx[:, ::-1].copy()
    perm_ring_k = P["ring_k"][:, :, :, ::-1].copy()
    perm_ring_v = P["ring_v"][:, :, :, ::-1].copy()
    W = P["ring_k"].shape[3]
    full = np.full_like(P["pos"], W)  # both sequences: all slots visible after reversal
    out = oracle.two_tier_attention(q, t1k, t1v, rev, P["ring_k"], P["ring_v"], P["pos"])
    np.testing.assert_allclose(out, base, rtol=1e-13, atol=1e-13)
    # sequence 1 is full: reversed slots hold the same tokens
    out = oracle.two_tier_attention(q, t1k, t1v, idx, perm_ring_k, perm_ring_v, full)
    np.testing.assert_allclose(out[1], base[1], rtol=1e-13, atol=1e-13)
    # default scale is 1/sqrt(d); an explicit scale s equals the query scaled by s*sqrt(d)
    d = q.shape[-1]
    s = 0.37
    out = oracle.two_tier_attention(q, t1k, t1v, idx, P["ring_k"], P["ring_v"], P["pos"], scale=s)
    out2 = oracle.two_tier_attention(q * s * math.sqrt(d), t1k, t1v, idx, P["ring_k"],
                                     P["ring_v"], P["pos"])
    np.testing.assert_allclose(out, out2, rtol=1e-12, atol=1e-12)


def test_new_token_attends_to_itself():
    B, L, Hq, Hkv, d, W = 1, 1, 2, 1, 4, 3
    rng = np.random.default_rng(71)
    ring_k = rng.standard_normal((B, L, Hkv, W, d))
    ring_v = rng.standard_normal((B, L, Hkv, W, d))
    pos = np.array([W], dtype=np.int64)
    kn = np.zeros((B, L, Hkv, d)); kn[..., 0] = 50.0
    vn = np.full((B, L, Hkv, d), 7.0)
    q = np.zeros((B, L, Hq, d)); q[..., 0] = 50.0
    out = oracle.decode_step(q, np.zeros((B, L, Hkv, 1, d)), np.zeros((B, L, Hkv, 1, d)),
                             None, ring_k, ring_v, pos, kn, vn, scale=1.0)
    np.testing.assert_allclose(out, 7.0, rtol=0, atol=1e-12)


def test_bf16_inputs_are_read_exactly():
    x = np.array([1.0, -2.5, 3.140625, 1e-3, -65504.0], dtype=np.float32)
    bits = f32_to_bf16_bits(x)
    t = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(oracle.bf16_to_f64(bits), t)


# ----------------------------------------------------------------------------
# Rotary position embedding of the GQA-layer decode step (decoders' RoPE)
# ----------------------------------------------------------------------------

def test_rope_closed_forms():
    # d = 2: one pair rotated by angle p (theta^0 = 1)
    for p in (0.0, 0.5, 3.0, 1000.0):
        np.testing.assert_allclose(oracle.rope_rotate(np.array([1.0, 0.0]), p, 10000.0),
                                   [math.cos(p), math.sin(p)], rtol=0, atol=1e-15)
        np.testing.assert_allclose(oracle.rope_rotate(np.array([0.0, 1.0]), p, 10000.0),
                                   [-math.sin(p), math.cos(p)], rtol=0, atol=1e-15)
    # angle of pair i is p * theta^(-2i/d): d = 128, theta = 10^4 -> pair 32 is p / 100
    a = oracle.rope_angles(128, 7.0, 10000.0)
    assert a[0] == 7.0 and a[32] == pytest.approx(0.07, rel=1e-14)
    assert a[63] == pytest.approx(7.0 * 10000.0 ** (-126 / 128), rel=1e-14)
    # position 0 is the identity
    x = np.random.default_rng(0).standard_normal((3, 64))
    np.testing.assert_array_equal(oracle.rope_rotate(x, 0, 500000.0), x)


def test_rope_matches_complex_rotation_of_half_split_pairs():
    """Independent formulation: z_i = x_i + 1j * x_{i + d/2} times e^{1j a_i}."""
    rng = np.random.default_rng(1)
    d, theta = 128, 500000.0
    x = rng.standard_normal((5, d))
    for p in (1, 17, 3639, 131071):
        i = np.arange(d // 2)
        z = (x[:, : d // 2] + 1j * x[:, d // 2:]) * np.exp(1j * p * theta ** (-2.0 * i / d))
        want = np.concatenate([z.real, z.imag], axis=1)
        np.testing.assert_allclose(oracle.rope_rotate(x, p, theta), want, rtol=0, atol=1e-12)


def test_rope_relative_position_and_composition():
    rng = np.random.default_rng(2)
    d, theta = 64, 10000.0
    q, k = rng.standard_normal(d), rng.standard_normal(d)
    for m, n in ((5, 3), (100, 7), (2000, 1999)):
        lhs = oracle.rope_rotate(q, m, theta) @ oracle.rope_rotate(k, n, theta)
        rhs = oracle.rope_rotate(q, m - n, theta) @ k
        assert lhs == pytest.approx(rhs, rel=1e-10, abs=1e-10)
    np.testing.assert_allclose(oracle.rope_rotate(oracle.rope_rotate(q, 30, theta), 12, theta),
                               oracle.rope_rotate(q, 42, theta), rtol=0, atol=1e-12)
    # rotation preserves every pair's length
    r = oracle.rope_rotate(q, 77, theta)
    np.testing.assert_allclose(r[: d // 2] ** 2 + r[d // 2:] ** 2,
                               q[: d // 2] ** 2 + q[d // 2:] ** 2, rtol=1e-12)


def test_f64_to_bf16_rounds_to_nearest_even():
    # values exactly representable in fp32: torch's fp32 -> bf16 cast is RNE
    rng = np.random.default_rng(3)
    x = rng.standard_normal(10000).astype(np.float32).astype(np.float64)
    want = torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16).view(torch.int16).numpy()
    np.testing.assert_array_equal(oracle.f64_to_bf16_bits(x), want.view(np.uint16))
    # exact midpoints between bf16 neighbours of 1: 1 + 2^-8 -> 1 (even), 1 + 3*2^-8 -> 1 + 2^-6
    got = oracle.f64_to_bf16_bits(np.array([1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -1.0 - 2.0 ** -8]))
    assert got.tolist() == [0x3F80, 0x3F82, 0xBF80]
    # a value just above a midpoint (not representable in fp32) rounds up
    assert oracle.f64_to_bf16_bits(np.array([1.0 + 2.0 ** -8 + 2.0 ** -40]))[0] == 0x3F81


def test_rope_step_at_position_zero_is_the_plain_step():
    w = WORKLOADS["tiny"].with_(B=2, W0=(0, 0), T=1)
    kv = kv_inputs(w)
    st = step_inputs(w, 0)
    idx = np.tile(np.arange(w.k), (w.B, 1))
    a = (kv.ring_k.copy(), kv.ring_v.copy(), kv.pos0.copy())
    b = (kv.ring_k.copy(), kv.ring_v.copy(), kv.pos0.copy())
    plain = oracle.decode_step(st.q, kv.tier1_k, kv.tier1_v, idx, *a, st.k_new, st.v_new)
    rope = oracle.decode_step_rope(st.q, kv.tier1_k, kv.tier1_v, idx, *b, st.k_new, st.v_new,
                                   theta=10000.0, rope_offset=0)
    np.testing.assert_array_equal(plain, rope)
    np.testing.assert_array_equal(a[0], b[0])


def test_rope_step_scores_depend_on_relative_positions():
    """Every key rotated at its own position and the query at the new
    token's: shifting all positions by the same amount leaves the output
    unchanged (the cache is built here, independently of the oracle's step)."""
    rng = np.random.default_rng(4)
    d, theta, n = 32, 10000.0, 9
    keys = rng.standard_normal((n, d))
    vals = rng.standard_normal((n, d))
    q = rng.standard_normal(d)
    outs = []
    for shift in (0, 250, 4000):
        K = np.stack([oracle.rope_rotate(keys[i], shift + i, theta) for i in range(n)])
        qr = oracle.rope_rotate(q, shift + n - 1, theta)
        outs.append(oracle.softmax_attention(qr, K, vals, 1 / math.sqrt(d)))
    np.testing.assert_allclose(outs[1], outs[0], rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(outs[2], outs[0], rtol=1e-10, atol=1e-12)


def test_rope_step_rotates_query_and_stored_key_at_offset_plus_pos():
    w = WORKLOADS["tiny"].with_(B=2, W0=(5, 128), T=1)
    kv = kv_inputs(w)
    st = step_inputs(w, 0)
    idx = np.tile(np.arange(w.k), (w.B, 1))
    rk, rv, pos = kv.ring_k.copy(), kv.ring_v.copy(), kv.pos0.copy()
    theta, off = 500000.0, w.k
    out = oracle.decode_step_rope(st.q, kv.tier1_k, kv.tier1_v, idx, rk, rv, pos, st.k_new,
                                  st.v_new, theta=theta, rope_offset=off)
    for b, p0 in enumerate(kv.pos0):
        slot = int(p0) % w.W
        # the stored key is the bf16 rounding of the rotated key; the value is unchanged
        want = oracle.f64_to_bf16_bits(oracle.rope_rotate(st.k_new[b], off + int(p0), theta))
        np.testing.assert_array_equal(rk[b, :, :, slot], want)
        np.testing.assert_array_equal(rv[b, :, :, slot], st.v_new[b])
        # query head 3 of layer 0 against torch SDPA on the assembled keys
        g = 3 // w.G
        K, V = oracle.two_tier_kv(kv.tier1_k, kv.tier1_v, idx[b], rk, rv, int(pos[b]), b, 0, g)
        qr = oracle.rope_rotate(st.q[b, 0, 3], off + int(p0), theta)
        ref = F.scaled_dot_product_attention(
            torch.from_numpy(qr)[None, None, None], torch.from_numpy(K)[None, None],
            torch.from_numpy(V)[None, None])[0, 0, 0].numpy()
        np.testing.assert_allclose(out[b, 0, 3], ref, rtol=1e-10, atol=1e-12)


# ----------------------------------------------------------------------------
# Question-side prologue: q_vec, CME-guided localisation, Tier-2 start
# ----------------------------------------------------------------------------

def test_question_vector_closed_forms():
    tok = np.zeros((3, 4, 2), dtype=np.float32)
    tok[0, :3] = [[1.0, 2.0], [1.0, 2.0], [1.0, 2.0]]   # constant rows -> that row
    tok[1, :2] = [[1.0, -3.0], [3.0, 5.0]]             # two rows -> their midpoint
    tok[0, 3] = tok[1, 2:] = np.nan                     # padding is never read
    q = oracle.question_vector(tok, np.array([3, 2, 0]))
    np.testing.assert_array_equal(q, [[1.0, 2.0], [2.0, 1.0], [0.0, 0.0]])


def test_question_vector_matches_torch_mean():
    rng = np.random.default_rng(5)
    tok = rng.standard_normal((4, 9, 33)).astype(np.float32)
    qlen = np.array([9, 1, 5, 7])
    q = oracle.question_vector(tok, qlen)
    for b in range(4):
        want = torch.from_numpy(tok[b, :qlen[b]]).double().mean(dim=0).numpy()
        np.testing.assert_allclose(q[b], want, rtol=1e-15, atol=1e-15)


def test_tier2_start_formula_cases():
    # start = max(0, min(|C| - W, alpha - W/2))
    assert oracle.tier2_start(100, 1000, 64) == 68
    assert oracle.tier2_start(10, 1000, 64) == 0        # clamped at the context start
    assert oracle.tier2_start(990, 1000, 64) == 936     # clamped so the window ends at |C|
    assert oracle.tier2_start(500, 40, 64) == 0         # context shorter than the window
    assert oracle.tier2_start(77, 1000, 63) == 46       # W/2 rounded down


def test_cme_locate_argmax_norm_and_ties():
    bank = np.zeros((2, 5, 3), dtype=np.float32)
    bank[0] = [[1, 0, 0], [0, 3, 0], [2, 0, 0], [0, 0, -2.5], [1, 1, 1]]   # norms 1,3,2,2.5,1.73
    bank[1] = [[0, 2, 0], [2, 0, 0], [0, 0, 2], [1, 1, 1], [0, 0, 0]]      # three rows tie at 2
    offs = np.array([[0, 256, 512, 768, 1024], [0, 10, 20, 30, 40]], dtype=np.int32)
    alpha, start, j = oracle.cme_locate(bank, offs, np.array([4096, 50]), 64)
    assert j.tolist() == [1, 0]                         # ties -> lower index
    assert alpha.tolist() == [256, 0]
    assert start.tolist() == [224, 0]
    # brute force on random banks: the row of largest Euclidean norm
    rng = np.random.default_rng(6)
    bank = rng.standard_normal((3, 50, 16)).astype(np.float32)
    _, _, j = oracle.cme_locate(bank, np.tile(np.arange(50, dtype=np.int32), (3, 1)),
                                np.full(3, 100), 8)
    for b in range(3):
        norms = [math.sqrt(sum(float(x) ** 2 for x in row)) for row in bank[b]]
        assert j[b] == max(range(50), key=lambda i: (norms[i], -i))


def test_cme_locate_decides_in_float32():
    # two squared norms that differ in fp64 but round to the same float32:
    # the decision is a tie and goes to the lower index
    bank = np.zeros((1, 2, 2), dtype=np.float32)
    bank[0, 0] = [1.0, 0.0]
    bank[0, 1] = [1.0, 2.0 ** -13]    # squared norm 1 + 2^-26 rounds to 1 in float32
    _, _, j = oracle.cme_locate(bank, np.zeros((1, 2), dtype=np.int32), np.array([10]), 4)
    assert j[0] == 0


def test_question_inputs_carry_the_planted_selection():
    """The generated tokens average to the planted question vector, so the
    selection of the pooled vector is the planted set (margin 2e-4)."""
    from workloads import question_inputs
    w = WORKLOADS["tiny"].with_(B=3)
    si = selection_inputs(w)
    qi = question_inputs(w, si)
    q, idx, _, alpha, start = oracle.question_select(qi.tokens, qi.q_len, si.cme_bank, w.k,
                                                     qi.chunk_offset, qi.ctx_len, w.W)
    np.testing.assert_allclose(q, si.question_emb, rtol=0, atol=1e-6)
    np.testing.assert_array_equal(idx, si.planted_idx)
    assert np.all((0 <= start) & (start <= qi.ctx_len - w.W))


# ----------------------------------------------------------------------------
# MemoryBridge output: LayerNorm, norm-calibrated tanh, norm cap (Section 2.2)
# ----------------------------------------------------------------------------

def test_bridge_epilogue_closed_forms():
    nu = 0.7
    # (a, -a): LayerNorm gives (a, -a)/sqrt(a^2 + eps); 1.077 nu < 2 nu: no cap
    a = 3.0
    z = a / math.sqrt(a * a + 1e-5)
    got = oracle.bridge_epilogue(np.array([[a, -a]]), np.ones(2), np.zeros(2), nu)
    np.testing.assert_allclose(got, [[nu * math.tanh(z), -nu * math.tanh(z)]], rtol=1e-14)
    # 16 features of +-a: ||nu tanh|| = 4 nu tanh(z) > 2 nu: scaled to norm 2 nu exactly
    x = np.array([[a, -a] * 8])
    got = oracle.bridge_epilogue(x, np.ones(16), np.zeros(16), nu)
    np.testing.assert_allclose(np.linalg.norm(got), 2 * nu, rtol=1e-14)
    np.testing.assert_allclose(got, 2 * nu * np.sign(x) / 4.0, rtol=1e-14)
    # a constant row has zero variance: LayerNorm gives beta; zero beta -> zero vector
    got = oracle.bridge_epilogue(np.full((1, 8), 5.0), np.ones(8), np.zeros(8), nu)
    np.testing.assert_array_equal(got, np.zeros((1, 8)))


def test_bridge_epilogue_against_torch_and_the_norm_bound():
    rng = np.random.default_rng(8)
    rows, D, nu = 37, 256, 0.9
    x = rng.standard_normal((rows, D)) * 3 + 1
    gamma = 1 + 0.1 * rng.standard_normal(D)
    beta = 0.1 * rng.standard_normal(D)
    ln = F.layer_norm(torch.from_numpy(x), (D,), torch.from_numpy(gamma), torch.from_numpy(beta),
                      eps=1e-5)
    t = nu * torch.tanh(ln)
    cap = torch.clamp(2 * nu / t.norm(dim=-1, keepdim=True), max=1.0)
    got = oracle.bridge_epilogue(x, gamma, beta, nu)
    np.testing.assert_allclose(got, (t * cap).numpy(), rtol=1e-12, atol=1e-14)
    norms = np.linalg.norm(got, axis=-1)
    assert np.all(norms <= 2 * nu * (1 + 1e-12))
    # rows under the cap are exactly nu tanh(LayerNorm(x)): shrink them below it
    small = oracle.bridge_epilogue(x, gamma * 0.01, beta * 0.01, nu)
    np.testing.assert_allclose(small, nu * np.tanh(F.layer_norm(
        torch.from_numpy(x), (D,), torch.from_numpy(gamma * 0.01),
        torch.from_numpy(beta * 0.01), eps=1e-5).numpy()), rtol=1e-12, atol=1e-15)


# ----------------------------------------------------------------------------
# Graph-based context denoising (Section 2.1; keep-minimum from the appendix)
# ----------------------------------------------------------------------------

def test_denoise_closed_forms():
    u, v = np.array([1.0, 0.0, 0.0]), np.array([0.0, 1.0, 0.0])
    w = np.array([1.0, 1.0, 0.0])               # cos(u, w) = cos(v, w) = 1/sqrt(2)
    e = np.stack([u, u, v, w, v, u, v])
    # g = 1: cos to the next token: 1, 0, .707, .707, 0, 0, (none)
    keep = oracle.denoise_keep(e, 7, 1, 0.5, 0)
    assert keep.tolist() == [True, False, True, True, False, False, False]
    # g = 2: token 1 sees v (0) and w (.707); token 4 sees u, v (0, 1); token 5 sees v (0)
    keep = oracle.denoise_keep(e, 7, 2, 0.5, 0)
    assert keep.tolist() == [True, True, True, True, True, False, False]
    # a zero vector has cosine 0 with everything
    e0 = np.stack([u, np.zeros(3), u])
    assert oracle.denoise_keep(e0, 3, 1, 0.0, 0).tolist() == [True, True, False]
    assert oracle.denoise_keep(e0, 3, 1, 0.1, 0).tolist() == [False, False, False]


def test_denoise_thresholds_at_the_extremes():
    rng = np.random.default_rng(12)
    e = rng.standard_normal((100, 8))
    # tau = -1: every token with a follower passes; the last has none
    keep = oracle.denoise_keep(e, 100, 3, -1.0, 16)
    assert keep.sum() == 99 and not keep[-1]
    # tau > 1: nothing passes; the keep-minimum alone keeps 15, 31, 47, ...
    keep = oracle.denoise_keep(e, 100, 3, 1.5, 16)
    assert np.flatnonzero(keep).tolist() == [15, 31, 47, 63, 79, 95]


def test_denoise_against_an_independent_formulation():
    """Threshold test from torch's pairwise cosines over shifted copies; the
    keep-minimum from its closed form: a token that fails the test is kept
    exactly when its distance to the last token that passed it (or to
    position -1) is a multiple of keep_every."""
    rng = np.random.default_rng(13)
    n, H, g, tau, every = 700, 16, 3, 0.35, 16
    steps = rng.standard_normal((n, H)) * 0.6
    steps[rng.random(n) < 0.3] *= 6.0              # isolated tokens
    e = np.cumsum(steps, axis=0)                    # neighbours correlate
    et = torch.from_numpy(e)
    best = torch.full((n,), -math.inf, dtype=torch.float64)
    for s in range(1, g + 1):
        c = F.cosine_similarity(et[:-s], et[s:], dim=1, eps=0.0)
        best[:-s] = torch.maximum(best[:-s], c)
    passed = (best >= tau).numpy()
    last, want = -1, np.zeros(n, dtype=bool)
    for i in range(n):
        want[i] = passed[i] or (i - last) % every == 0
        if passed[i]:
            last = i
    got = oracle.denoise_keep(e, n, g, tau, every)
    np.testing.assert_array_equal(got, want)
    kept = np.flatnonzero(got)
    assert np.all(np.diff(np.concatenate([[-1], kept])) <= every)   # no gap above 16
    assert 0 < kept.size < n
    idx, cnt = oracle.denoise(e[None], np.array([n]), g, tau, every)
    assert cnt[0] == kept.size and idx[0, :kept.size].tolist() == kept.tolist()
    assert np.all(idx[0, kept.size:] == -1)
