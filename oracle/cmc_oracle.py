"""Plain, slow fp64 CPU oracle of the CMC two-tier decode path.

TEST INFRASTRUCTURE ONLY.  Nothing in the product imports this module; the
CUDA library never calls it and it never calls the CUDA library.

What it computes, following Section 2.5 of the paper ("Inference with Two-Tier
KV Cache Policy"):

* Tier-1 scoring: the cosine similarity between each decoder-ready CME m_j and
  the mean-pooled question vector q_vec (the score_j equation of Section 2.5).
* Tier-1 selection: keep the K highest-scoring CMEs, then re-order the kept
  ones by original document position, i.e. by ascending index (Section 2.5,
  text after the score_j equation).
* Tier-2 window: a ring of W token slots per (sequence, layer, KV head) that
  receives each generated token; the cache then stays bounded by K + W + |q|
  tokens at every generation step (Section 2.5, "KV cache assembly").
* Decode attention: for each query head, softmax(q . k_i * scale) over the
  keys of [Tier-1 | Tier-2], applied to the values.  The MAC model of the
  appendix ("Attention MACs Analysis", MACs_t = 2 n_h d_h n_l L_t) counts
  exactly this per-step work over L_t cached keys.

Readings where the paper is silent (each is also listed in the design notes):

* A zero vector has no direction; its cosine score is taken as 0.
* Ties in score go to the lower index, and the selection decision is taken on
  the scores rounded to float32, the precision the kernels compute them in.
  Scores themselves are computed in fp64.
* The ring slot of token number p (counting from 0) is p mod W; once more than
  W tokens have been appended the oldest is overwritten (sliding window).
* Within a decode step the new token is appended before attention, so it
  attends to itself (standard autoregressive decoding).
* scale defaults to 1/sqrt(d); cached keys are taken as already position-
  encoded, so no rotary embedding is applied here; nothing is masked.
* Query head h reads KV head h // (Hq / Hkv) (grouped-query attention).
* An empty cache (no Tier-1 rows and no ring tokens) yields a zero output.
* The decode step of a real GQA layer (decode_step_rope) rotates the new
  query and key with rotary position embedding, which the paper's decoders
  apply but the paper does not restate; its readings are listed above that
  function.

Parity status: every function here is pinned by the tests in
tests/test_oracle_pins.py (closed forms, brute force, library routines,
invariants); none is "parity unpinned".
"""

from __future__ import annotations

import math
from typing import Iterable, Optional, Tuple

import numpy as np


# ----------------------------------------------------------------------------
# Inputs
# ----------------------------------------------------------------------------

def bf16_to_f64(a: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> float64, exact.  Float arrays pass
    through as float64."""
    a = np.asarray(a)
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)
    return a.astype(np.float64)


# ----------------------------------------------------------------------------
# Tier-1: question-guided scoring and top-K selection (Section 2.5)
# ----------------------------------------------------------------------------

def cosine_scores(question_emb: np.ndarray, cme_bank: np.ndarray) -> np.ndarray:
    """score[b, j] = (m_j . q_vec) / (||m_j|| ||q_vec||)  (Section 2.5, score_j).

    question_emb: [B, D]; cme_bank: [B, N, D].  Returns float64 [B, N].
    A zero-norm CME or question vector gives score 0.
    """
    q = np.asarray(question_emb, dtype=np.float64)
    m = np.asarray(cme_bank)
    B, N, D = m.shape
    out = np.zeros((B, N), dtype=np.float64)
    for b in range(B):
        qn = math.sqrt(float(q[b] @ q[b]))
        for j0 in range(0, N, 4096):
            rows = m[b, j0:j0 + 4096].astype(np.float64)
            dots = rows @ q[b]
            mn = np.sqrt(np.einsum("ij,ij->i", rows, rows))
            den = mn * qn
            s = np.zeros_like(dots)
            nz = den > 0.0
            s[nz] = dots[nz] / den[nz]
            out[b, j0:j0 + 4096] = s
    return out


def select_top_k(scores: np.ndarray, k: int) -> np.ndarray:
    """The k highest scores per row, returned as indices in ascending order
    (Section 2.5: top-K, then re-ordered by original document position).

    The decision is taken on the scores rounded to float32; equal scores go to
    the lower index.  Returns int64 [B, k].
    """
    s = np.asarray(scores)
    B, N = s.shape
    if not 0 <= k <= N:
        raise ValueError(f"k={k} outside [0, N={N}]")
    s32 = s.astype(np.float32)
    out = np.empty((B, k), dtype=np.int64)
    j = np.arange(N)
    for b in range(B):
        # primary key: score descending; secondary: index ascending
        ranked = np.lexsort((j, -s32[b]))
        out[b] = np.sort(ranked[:k])
    return out


def score_select(question_emb: np.ndarray, cme_bank: np.ndarray, k: int
                 ) -> Tuple[np.ndarray, np.ndarray]:
    """Tier-1 selection M* = TopK(M, q, K) (Section 2.5).  Returns (idx, scores)."""
    scores = cosine_scores(question_emb, cme_bank)
    return select_top_k(scores, k), scores


# ----------------------------------------------------------------------------
# Graph-based context denoising (Section 2.1)
# ----------------------------------------------------------------------------

def denoise_pass(emb: np.ndarray, n_tokens: int, g: int, tau: float) -> np.ndarray:
    """The threshold test of the graph-based denoising (Section 2.1): token i
    passes when its cosine similarity to at least one of its g following
    tokens (j = i+1 .. min(i+g, n)) is at least tau; the last token has no
    follower and fails.  Cosines of zero vectors are 0; the comparison with
    tau is taken on the cosine rounded to float32 (the kernels' precision).
    emb: [>= n_tokens, H].  Returns bool [n_tokens]."""
    e = np.asarray(emb[:n_tokens], dtype=np.float64)
    n = e.shape[0]
    norms = np.sqrt(np.einsum("ij,ij->i", e, e))
    passed = np.zeros(n, dtype=bool)
    for i in range(n):
        best = -np.inf
        for j in range(i + 1, min(i + g, n - 1) + 1):
            den = norms[i] * norms[j]
            c = float(e[i] @ e[j]) / den if den > 0 else 0.0
            best = max(best, c)
        passed[i] = bool(np.float32(best) >= np.float32(tau))
    return passed


def keep_minimum(passed: np.ndarray, keep_every: int) -> np.ndarray:
    """The keep-minimum constraint of the threshold appendix: one kept token
    in every run of `keep_every` consecutive positions.  Walking left to
    right, a token is also kept when the previous kept token lies
    `keep_every` positions back (or, before any, when it is token
    keep_every - 1); keep_every == 0 keeps just the passing tokens."""
    keep = np.array(passed, dtype=bool)
    last = -1
    for i in range(keep.size):
        if not keep[i] and keep_every > 0 and i - last >= keep_every:
            keep[i] = True
        if keep[i]:
            last = i
    return keep


def denoise_keep(emb: np.ndarray, n_tokens: int, g: int, tau: float, keep_every: int
                 ) -> np.ndarray:
    """Which tokens of one context survive the denoising: the threshold test
    followed by the keep-minimum.  Returns bool [n_tokens]."""
    return keep_minimum(denoise_pass(emb, n_tokens, g, tau), keep_every)


def denoise(emb: np.ndarray, n_tokens: np.ndarray, g: int, tau: float, keep_every: int
            ) -> Tuple[np.ndarray, np.ndarray]:
    """Denoised contexts as index lists: for each context b, the positions of
    the kept tokens in ascending order (int64 [B, max_n], -1 past the count)
    and the counts (int64 [B])."""
    emb = np.asarray(emb)
    B, n_max = emb.shape[0], emb.shape[1]
    idx = np.full((B, n_max), -1, dtype=np.int64)
    cnt = np.zeros(B, dtype=np.int64)
    for b in range(B):
        kept = np.flatnonzero(denoise_keep(emb[b], int(n_tokens[b]), g, tau, keep_every))
        idx[b, :len(kept)] = kept
        cnt[b] = len(kept)
    return idx, cnt


# ----------------------------------------------------------------------------
# MemoryBridge output (Section 2.2, the norm-calibrated tanh equation)
# ----------------------------------------------------------------------------

def bridge_epilogue(x: np.ndarray, gamma: np.ndarray, beta: np.ndarray, nu: float,
                    eps: float = 1e-5) -> np.ndarray:
    """The decoder-ready CMEs from the MemoryBridge MLP output x [rows, H_d]:
    m_hat = LayerNorm(x) (mean and biased variance over the features, eps,
    per-feature gamma and beta: PyTorch's default, as the hyperparameter
    appendix states), then m = nu tanh(m_hat) min(1, 2 nu / ||nu tanh(m_hat)||)
    (Section 2.2), so that ||m|| <= 2 nu.  Returns fp64 [rows, H_d]."""
    x = np.asarray(x, dtype=np.float64)
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    m_hat = np.asarray(gamma, np.float64) * (x - mu) / np.sqrt(var + eps) + np.asarray(beta, np.float64)
    t = nu * np.tanh(m_hat)
    n = np.sqrt((t * t).sum(axis=-1, keepdims=True))
    with np.errstate(divide="ignore"):
        f = np.minimum(1.0, np.where(n > 0, 2.0 * nu / n, np.inf))
    return t * f


# ----------------------------------------------------------------------------
# Question-side prologue (Section 2.5 and the appendix on localisation
# without annotations)
# ----------------------------------------------------------------------------

def question_vector(tokens: np.ndarray, q_len: np.ndarray) -> np.ndarray:
    """q_vec: the mean of the question tokens' input embeddings (Section 2.5,
    Tier-1).  tokens: [B, Lq, D]; q_len: [B] tokens per question (rows past it
    are ignored; an empty question gives the zero vector).  Returns fp64
    [B, D]."""
    tokens = np.asarray(tokens)
    B, _, D = tokens.shape
    out = np.zeros((B, D), dtype=np.float64)
    for b in range(B):
        n = int(q_len[b])
        if n > 0:
            out[b] = tokens[b, :n].astype(np.float64).sum(axis=0) / n
    return out


def tier2_start(alpha: int, ctx_len: int, W: int) -> int:
    """Start of the W-token local window centred on alpha (Section 2.5,
    Tier-2): max(0, min(|C| - W, alpha - W/2)), W/2 rounded down."""
    return max(0, min(int(ctx_len) - W, int(alpha) - W // 2))


def cme_locate(cme_bank: np.ndarray, chunk_offset: np.ndarray, ctx_len: np.ndarray, W: int
               ) -> Tuple[np.ndarray, np.ndarray, np.ndarray]:
    """CME-guided localisation (appendix on deployment without annotations):
    alpha = offset of the chunk that produced the highest-norm CME, and the
    Tier-2 start derived from it.  The argmax is decided on the squared norms
    rounded to float32 (the kernels' precision); equal norms go to the lower
    index.  Returns (alpha [B], start [B], j_max [B]) as int64."""
    m = np.asarray(cme_bank)
    B, N, D = m.shape
    alpha = np.empty(B, dtype=np.int64)
    start = np.empty(B, dtype=np.int64)
    jmax = np.empty(B, dtype=np.int64)
    for b in range(B):
        sq = np.empty(N, dtype=np.float64)
        for j0 in range(0, N, 4096):
            rows = m[b, j0:j0 + 4096].astype(np.float64)
            sq[j0:j0 + 4096] = np.einsum("ij,ij->i", rows, rows)
        sq32 = sq.astype(np.float32)
        j = int(np.flatnonzero(sq32 == sq32.max())[0])
        jmax[b] = j
        alpha[b] = int(chunk_offset[b, j])
        start[b] = tier2_start(alpha[b], ctx_len[b], W)
    return alpha, start, jmax


def question_select(tokens, q_len, cme_bank, k: int, chunk_offset, ctx_len, W: int):
    """The question-side prologue: q_vec, the Tier-1 selection and the Tier-2
    window start.  Returns (q_vec, idx, scores, alpha, start)."""
    q = question_vector(tokens, q_len)
    idx, scores = score_select(q, cme_bank, k)
    alpha, start, _ = cme_locate(cme_bank, chunk_offset, ctx_len, W)
    return q, idx, scores, alpha, start


# ----------------------------------------------------------------------------
# Tier-2: local-window ring (Section 2.5, Tier-2 and KV cache assembly)
# ----------------------------------------------------------------------------

def window_slots(pos: int, W: int) -> range:
    """Ring slots that hold tokens after `pos` tokens have been appended."""
    return range(min(int(pos), W))


def window_append(ring_k: np.ndarray, ring_v: np.ndarray, pos: np.ndarray,
                  k_new: np.ndarray, v_new: np.ndarray) -> None:
    """Append one token per sequence, in place.

    ring_k/ring_v: [B, L, Hkv, W, d]; pos: int64 [B] tokens appended so far;
    k_new/v_new: [B, L, Hkv, d].  Token number pos[b] goes to slot pos[b] mod W,
    overwriting the oldest token once the ring is full; pos[b] then grows by 1.
    """
    W = ring_k.shape[3]
    for b in range(ring_k.shape[0]):
        s = int(pos[b]) % W
        ring_k[b, :, :, s, :] = k_new[b]
        ring_v[b, :, :, s, :] = v_new[b]
        pos[b] += 1


# ----------------------------------------------------------------------------
# Decode attention over [Tier-1 | Tier-2]
# ----------------------------------------------------------------------------

def default_scale(d: int) -> float:
    return 1.0 / math.sqrt(d)


def softmax_attention(q: np.ndarray, K: np.ndarray, V: np.ndarray, scale: float
                      ) -> np.ndarray:
    """sum_i softmax_i(scale * q . k_i) v_i for one query vector, in fp64.

    q: [d]; K, V: [n, d].  n == 0 gives zeros.
    """
    q = np.asarray(q, dtype=np.float64)
    if K.shape[0] == 0:
        return np.zeros(V.shape[1], dtype=np.float64)
    z = scale * (np.asarray(K, dtype=np.float64) @ q)
    z = z - z.max()
    p = np.exp(z)
    return (p @ np.asarray(V, dtype=np.float64)) / p.sum()


def two_tier_kv(tier1_k, tier1_v, idx_b: Iterable[int], ring_k, ring_v, pos_b: int,
                b: int, l: int, g: int) -> Tuple[np.ndarray, np.ndarray]:
    """Keys and values one KV head sees: the Tier-1 bank rows at the selected
    indices, followed by the ring's occupied slots.  Returned as fp64 [n, d]."""
    sel = np.asarray(list(idx_b), dtype=np.int64)
    W = ring_k.shape[3]
    slots = np.asarray(window_slots(pos_b, W), dtype=np.int64)
    K = np.concatenate([bf16_to_f64(tier1_k[b, l, g][sel]),
                        bf16_to_f64(ring_k[b, l, g][slots])], axis=0)
    V = np.concatenate([bf16_to_f64(tier1_v[b, l, g][sel]),
                        bf16_to_f64(ring_v[b, l, g][slots])], axis=0)
    return K, V


def two_tier_attention_head(q, tier1_k, tier1_v, idx, ring_k, ring_v, pos,
                            b: int, l: int, h: int, scale: Optional[float] = None
                            ) -> np.ndarray:
    """Output of query head h of layer l, sequence b: fp64 [d]."""
    Hq = q.shape[2]
    Hkv = ring_k.shape[2]
    g = h // (Hq // Hkv)
    d = q.shape[3]
    sc = default_scale(d) if scale is None else scale
    idx_b = [] if idx is None else idx[b]
    K, V = two_tier_kv(tier1_k, tier1_v, idx_b, ring_k, ring_v, int(pos[b]), b, l, g)
    return softmax_attention(bf16_to_f64(q[b, l, h]), K, V, sc)


def two_tier_attention(q, tier1_k, tier1_v, idx, ring_k, ring_v, pos,
                       scale: Optional[float] = None) -> np.ndarray:
    """Decode attention over [Tier-1 | Tier-2] for every (b, l, h).

    q: [B, L, Hq, d]; tier1_k/v: [B, L, Hkv, N, d]; idx: [B, k] (or None for
    k = 0); ring_k/v: [B, L, Hkv, W, d]; pos: [B] tokens appended so far.
    Returns fp64 [B, L, Hq, d].
    """
    B, L, Hq, d = q.shape
    out = np.zeros((B, L, Hq, d), dtype=np.float64)
    for b in range(B):
        for l in range(L):
            for h in range(Hq):
                out[b, l, h] = two_tier_attention_head(
                    q, tier1_k, tier1_v, idx, ring_k, ring_v, pos, b, l, h, scale)
    return out


def decode_step(q, tier1_k, tier1_v, idx, ring_k, ring_v, pos, k_new, v_new,
                scale: Optional[float] = None) -> np.ndarray:
    """One decode step: append the new token to the ring, then attend.
    ring_k, ring_v and pos are updated in place."""
    window_append(ring_k, ring_v, pos, k_new, v_new)
    return two_tier_attention(q, tier1_k, tier1_v, idx, ring_k, ring_v, pos, scale)


# ----------------------------------------------------------------------------
# Decode step of a real GQA layer: rotary position embedding, then the step
# ----------------------------------------------------------------------------
#
# The paper runs frozen HuggingFace decoders (Llama-3, Mistral), which apply
# rotary position embedding (RoPE) to queries and keys and cache the rotated
# keys; it does not restate RoPE.  Readings used here:
#   * the half-split pairing of those implementations: element i is paired
#     with element i + d/2 and the pair is rotated by the angle
#     p * theta^(-2i/d), i < d/2;
#   * positions continue after the prefill input [M* || C_local || q]
#     ("KV cache assembly"): the token appended as number pos[b] of the ring
#     sits at position rope_offset + pos[b], where rope_offset counts the
#     positions before the ring (k, the Tier-1 rows);
#   * the rotated key is stored in the cache in bf16 (round to nearest even);
#     the query is used unrounded.

def rope_angles(d: int, p: float, theta: float) -> np.ndarray:
    """Rotation angle of each of the d/2 pairs at position p: p * theta^(-2i/d)."""
    i = np.arange(d // 2, dtype=np.float64)
    return float(p) * np.power(float(theta), -2.0 * i / d)


def rope_rotate(x: np.ndarray, p: float, theta: float) -> np.ndarray:
    """Rotate the last axis of x (fp64 or bf16 bits) by position p: the pair
    (x_i, x_{i+d/2}) becomes (x_i cos a_i - x_{i+d/2} sin a_i,
    x_{i+d/2} cos a_i + x_i sin a_i).  Returns fp64."""
    x = bf16_to_f64(x)
    d = x.shape[-1]
    a = rope_angles(d, p, theta)
    c, s = np.cos(a), np.sin(a)
    x1, x2 = x[..., : d // 2], x[..., d // 2:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def f64_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp64 -> bf16 bit patterns, rounding to nearest even in one step (the
    8 significant bits of bf16; finite values in bf16 range)."""
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)                         # x = m 2^e, 0.5 <= |m| < 1
    y = np.ldexp(np.round(m * 256.0) / 256.0, e)  # np.round: half to even
    return (y.astype(np.float32).view(np.uint32) >> np.uint32(16)).astype(np.uint16)


def decode_step_rope(q, tier1_k, tier1_v, idx, ring_k, ring_v, pos, k_new, v_new,
                     theta: float, rope_offset: int, scale: Optional[float] = None
                     ) -> np.ndarray:
    """One decode step of a GQA layer with rotary position embedding.

    q: [B, L, Hq, d] and k_new: [B, L, Hkv, d] are taken before rotation.  For
    each sequence, position p = rope_offset + pos[b] (pos before the append):
    the rotated key (bf16) and the value are appended to the ring, then the
    rotated query attends over [Tier-1 | Tier-2].  ring_k, ring_v and pos are
    updated in place.  Returns fp64 [B, L, Hq, d]."""
    B = q.shape[0]
    q_rot = np.empty(q.shape, dtype=np.float64)
    k_rot = np.empty(np.shape(k_new), dtype=np.uint16)
    for b in range(B):
        p = rope_offset + int(pos[b])
        q_rot[b] = rope_rotate(q[b], p, theta)
        k_rot[b] = f64_to_bf16_bits(rope_rotate(k_new[b], p, theta))
    window_append(ring_k, ring_v, pos, k_rot, v_new)
    return two_tier_attention(q_rot, tier1_k, tier1_v, idx, ring_k, ring_v, pos, scale)
