"""Seeded generation of the synthetic inputs.

Every tensor comes from its own counter-style numpy stream keyed by
(seed, tensor tag, sequence or step, attempt), so a slice of a workload (one
sequence, one decode step) can be regenerated without generating the rest.

bf16 tensors are returned as their raw 16-bit patterns (numpy uint16), rounded
to nearest-even from float32; both the CUDA path and the oracle read those same
bits.

Planted selection margin
------------------------
Bit-exact top-k parity needs a clear gap between the k-th and (k+1)-th cosine
score.  With i.i.d. Gaussian CMEs the natural gap at the cut is often below
1e-4 (at 16,384 rows it is about 5e-6), so rejection sampling alone cannot
meet that bar.  The bank is therefore built from prescribed cosines: each row
m_j keeps the norm and the q-orthogonal direction of a Gaussian draw g_j and
gets a component along q_vec chosen so that cos(m_j, q_vec) equals a target
c_j.  The targets are N(0, 1/D) draws (the spread of the cosine between random
directions in D dimensions); the k largest are raised by `margin` and the
targets are then assigned to rows by a random permutation, so the k rows that
received the raised targets (`planted_idx`) are the top-k by construction,
with a gap of at least `margin` before float32 rounding.  Rounding the rows to
float32 moves a cosine by ~1e-7, far below the margin.
"""

from __future__ import annotations

from dataclasses import dataclass
from typing import Optional

import numpy as np

from .configs import Workload

_TAGS = {
    "question": 1,
    "cosines": 2,
    "perm": 3,
    "bank": 4,
    "tier1_k": 5,
    "tier1_v": 6,
    "ring_k": 7,
    "ring_v": 8,
    "step_q": 9,
    "step_k": 10,
    "step_v": 11,
    "idx": 12,
    "question_tokens": 13,
    "context_vocab": 14,
    "context_ids": 15,
}


def _rng(seed: int, tag: str, *extra: int) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence([seed, _TAGS[tag], *extra]))


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns (uint16), round to nearest even.

    Inputs are finite, so the NaN path of a full conversion is not needed."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = ((u >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((u + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> float32, exact."""
    return (np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32)
            << np.uint32(16)).view(np.float32)


def _torch_gen(seed: int, tag: str, *extra: int):
    import torch
    s = np.random.SeedSequence([seed, _TAGS[tag], *extra]).generate_state(1, np.uint64)[0]
    return torch.Generator().manual_seed(int(s) & 0x7FFFFFFFFFFFFFFF)


def _gauss_bf16(key, shape, std: float) -> np.ndarray:
    """Gaussian bf16 bit patterns; torch's float32 -> bfloat16 cast rounds to
    nearest even, like f32_to_bf16_bits."""
    import torch
    x = torch.randn(tuple(shape), generator=_torch_gen(*key), dtype=torch.float32)
    x.mul_(float(std))
    return x.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


# ----------------------------------------------------------------------------
# Tier-1 selection inputs: question vector and CME bank
# ----------------------------------------------------------------------------

@dataclass
class SelectionInputs:
    question_emb: np.ndarray  # float32 [B, D]
    cme_bank: np.ndarray  # float32 [B, N, D]
    planted_idx: Optional[np.ndarray]  # int64 [B, k] ascending, when a margin was planted


def _target_cosines(w: Workload, b: int, attempt: int):
    rng = _rng(w.seed, "cosines", b, attempt)
    c = rng.standard_normal(w.N) / np.sqrt(w.D)
    c = np.clip(c, -0.95, 0.95)
    planted = None
    if w.margin > 0 and 0 < w.k < w.N:
        order = np.argsort(-c, kind="stable")
        ranked = c[order]
        ranked[: w.k] += w.margin
        perm = _rng(w.seed, "perm", b, attempt).permutation(w.N)
        c = np.empty_like(ranked)
        c[perm] = ranked
        planted = np.sort(perm[: w.k]).astype(np.int64)
    return c, planted


def _bank_rows(w: Workload, b: int, attempt: int, qhat: np.ndarray, c: np.ndarray,
               out: np.ndarray, chunk: int = 2048) -> None:
    import torch
    qh = torch.from_numpy(qhat)
    out_t = torch.from_numpy(out)
    work = torch.empty((min(chunk, w.N), w.D), dtype=torch.float64)
    for r0 in range(0, w.N, chunk):
        r1 = min(w.N, r0 + chunk)
        g = work[: r1 - r0]
        g.copy_(torch.randn((r1 - r0, w.D), generator=_torch_gen(w.seed, "bank", b, attempt, r0),
                            dtype=torch.float32))
        g.mul_(float(w.emb_std))
        # g = along * qhat + perp with perp orthogonal to qhat; the row keeps
        # |g| and the direction of perp, and gets cosine c_j with q:
        #   m = |g| (c_j qhat + sqrt(1 - c_j^2) perp / |perp|)
        along = g @ qh
        rho2 = torch.linalg.vector_norm(g, dim=1) ** 2
        rho = rho2.sqrt()
        pn = (rho2 - along * along).sqrt()
        cj = torch.from_numpy(np.ascontiguousarray(c[r0:r1]))
        coef_perp = rho * (1.0 - cj * cj).sqrt() / pn
        coef_q = rho * cj - coef_perp * along
        g.mul_(coef_perp[:, None])
        g.addr_(coef_q, qh)
        out_t[r0:r1].copy_(g)


def selection_inputs(w: Workload, attempt: int = 0, batch: Optional[range] = None
                     ) -> SelectionInputs:
    """Question vectors and CME banks for sequences `batch` (default: all B)."""
    seqs = range(w.B) if batch is None else batch
    nb = len(seqs)
    q_out = np.empty((nb, w.D), dtype=np.float32)
    bank = np.empty((nb, w.N, w.D), dtype=np.float32)
    planted = [] if (w.margin > 0 and 0 < w.k < w.N) else None
    for i, b in enumerate(seqs):
        q = _rng(w.seed, "question", b, attempt).standard_normal(w.D) * w.emb_std
        q32 = q.astype(np.float32)
        q64 = q32.astype(np.float64)
        qhat = q64 / np.sqrt(q64 @ q64)
        c, pl = _target_cosines(w, b, attempt)
        _bank_rows(w, b, attempt, qhat, c, bank[i])
        q_out[i] = q32
        if planted is not None:
            planted.append(pl)
    return SelectionInputs(
        question_emb=q_out, cme_bank=bank,
        planted_idx=None if planted is None else np.stack(planted),
    )


@dataclass
class QuestionInputs:
    tokens: np.ndarray        # float32 [B, Lq, D]: input embeddings of the question tokens
    q_len: np.ndarray         # int32 [B]: tokens of each question (rows past it are padding)
    chunk_offset: np.ndarray  # int32 [B, N]: context position of the chunk behind CME j
    ctx_len: np.ndarray       # int32 [B]: context length |C| in tokens


def question_inputs(w: Workload, si: SelectionInputs, Lq: int = 24, chunk: int = 256,
                    ratio: int = 4, batch: Optional[range] = None) -> QuestionInputs:
    """Question-side inputs around the question vectors of `si`.

    Each question has q_len tokens (24, 22, 20, ... ragged across sequences):
    the planted question vector plus noise of zero mean, so that the tokens'
    mean is that vector and the planted top-k margin carries over; padding
    rows hold other noise.  The context is cut into chunks of `chunk` tokens,
    each giving chunk / ratio consecutive CMEs, so CME j comes from the chunk
    at (j // (chunk / ratio)) * chunk and |C| = N * ratio."""
    seqs = range(w.B) if batch is None else batch
    nb = len(seqs)
    tokens = np.empty((nb, Lq, w.D), dtype=np.float32)
    q_len = np.empty(nb, dtype=np.int32)
    per_chunk = chunk // ratio
    offs = ((np.arange(w.N) // per_chunk) * chunk).astype(np.int32)
    for i, b in enumerate(seqs):
        n = max(1, Lq - 2 * (b % 5))
        rng = _rng(w.seed, "question_tokens", b)
        noise = rng.standard_normal((n, w.D)) * w.emb_std
        noise -= noise.mean(axis=0)
        tokens[i, :n] = (si.question_emb[i].astype(np.float64) + noise).astype(np.float32)
        tokens[i, n:] = (rng.standard_normal((Lq - n, w.D)) * w.emb_std).astype(np.float32)
        q_len[i] = n
    return QuestionInputs(tokens=tokens, q_len=q_len,
                          chunk_offset=np.tile(offs, (nb, 1)),
                          ctx_len=np.full(nb, w.N * ratio, dtype=np.int32))


@dataclass
class ContextInputs:
    emb: np.ndarray       # float32 [B, n, H]: input embeddings of the context tokens
    n_tokens: np.ndarray  # int32 [B]: tokens per context (rows past it are padding)


def context_inputs(w: Workload, H: int = 1280, ratio: int = 4, vocab: int = 4096,
                   batch: Optional[range] = None) -> ContextInputs:
    """Context token embeddings for the denoising filter: |C| = N * ratio
    tokens per context (the last context of a batch is 3/4 as long), each the
    embedding of a token id drawn with Zipf-like frequencies (p ~ 1/rank)
    from a vocabulary of independent Gaussian vectors, so that distinct
    tokens are nearly orthogonal and repeats of frequent tokens are close."""
    seqs = range(w.B) if batch is None else batch
    nb = len(seqs)
    n = w.N * ratio
    table = (_rng(w.seed, "context_vocab").standard_normal((vocab, H)) / np.sqrt(H)
             ).astype(np.float32)
    p = 1.0 / np.arange(1, vocab + 1)
    p /= p.sum()
    emb = np.zeros((nb, n, H), dtype=np.float32)
    n_tok = np.empty(nb, dtype=np.int32)
    for i, b in enumerate(seqs):
        nt = n if b + 1 < w.B or w.B == 1 else (3 * n) // 4
        ids = _rng(w.seed, "context_ids", b).choice(vocab, size=nt, p=p)
        emb[i, :nt] = table[ids]
        n_tok[i] = nt
    return ContextInputs(emb=emb, n_tokens=n_tok)


# ----------------------------------------------------------------------------
# Tier-1 K/V bank and Tier-2 ring
# ----------------------------------------------------------------------------

@dataclass
class KVInputs:
    tier1_k: np.ndarray  # bf16 bits [B, L, Hkv, N, d]
    tier1_v: np.ndarray  # bf16 bits [B, L, Hkv, N, d]
    ring_k: np.ndarray  # bf16 bits [B, L, Hkv, W, d]; slots >= fill are zero
    ring_v: np.ndarray  # bf16 bits [B, L, Hkv, W, d]
    pos0: np.ndarray  # int64 [B]: tokens appended so far (= fill before step 0)


def kv_inputs(w: Workload, batch: Optional[range] = None) -> KVInputs:
    seqs = range(w.B) if batch is None else batch
    nb = len(seqs)
    fill = w.fill()
    shp_bank = (w.L, w.Hkv, w.N, w.d)
    t1k = np.empty((nb,) + shp_bank, dtype=np.uint16)
    t1v = np.empty((nb,) + shp_bank, dtype=np.uint16)
    rk = np.zeros((nb, w.L, w.Hkv, w.W, w.d), dtype=np.uint16)
    rv = np.zeros((nb, w.L, w.Hkv, w.W, w.d), dtype=np.uint16)
    pos0 = np.empty(nb, dtype=np.int64)
    for i, b in enumerate(seqs):
        t1k[i] = _gauss_bf16((w.seed, "tier1_k", b), shp_bank, w.kv_std)
        t1v[i] = _gauss_bf16((w.seed, "tier1_v", b), shp_bank, w.kv_std)
        f = fill[b]
        assert 0 <= f <= w.W
        shp_ring = (w.L, w.Hkv, f, w.d)
        rk[i, :, :, :f] = _gauss_bf16((w.seed, "ring_k", b), shp_ring, w.kv_std)
        rv[i, :, :, :f] = _gauss_bf16((w.seed, "ring_v", b), shp_ring, w.kv_std)
        pos0[i] = f
    return KVInputs(t1k, t1v, rk, rv, pos0)


# ----------------------------------------------------------------------------
# Per-decode-step inputs
# ----------------------------------------------------------------------------

@dataclass
class StepInputs:
    q: np.ndarray  # bf16 bits [B, L, Hq, d]
    k_new: np.ndarray  # bf16 bits [B, L, Hkv, d]
    v_new: np.ndarray  # bf16 bits [B, L, Hkv, d]


def step_inputs(w: Workload, t: int, q_std: Optional[float] = None,
                parts: str = "qkv") -> StepInputs:
    """Query and new-token K/V of decode step t (all sequences, all layers).
    `parts` picks which of q, k_new, v_new to draw (the others are None)."""
    qs = w.q_std if q_std is None else q_std
    return StepInputs(
        q=_gauss_bf16((w.seed, "step_q", t), (w.B, w.L, w.Hq, w.d), qs)
        if "q" in parts else None,
        k_new=_gauss_bf16((w.seed, "step_k", t), (w.B, w.L, w.Hkv, w.d), w.kv_std)
        if "k" in parts else None,
        v_new=_gauss_bf16((w.seed, "step_v", t), (w.B, w.L, w.Hkv, w.d), w.kv_std)
        if "v" in parts else None,
    )


def random_tier1_indices(w: Workload, batch: Optional[range] = None) -> np.ndarray:
    """A seeded, ascending k-subset of [0, N) per sequence: int32 [B, k].

    Stands in for a selection result when the attention path is exercised
    without generating the CME bank."""
    seqs = range(w.B) if batch is None else batch
    out = np.empty((len(seqs), w.k), dtype=np.int32)
    for i, b in enumerate(seqs):
        rng = _rng(w.seed, "idx", b)
        out[i] = np.sort(rng.choice(w.N, size=w.k, replace=False))
    return out
