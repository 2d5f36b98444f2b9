"""The synthetic workloads of the CMC two-tier decode path.

Each workload fixes the shapes of one decode problem:

* the Tier-1 side: a bank of N Context Memory Embeddings (CMEs) of dimension D
  per sequence, a question vector q_vec of dimension D, and a top-K budget k
  (Section 2.5, "Tier-1: question-guided top-K selection");
* per layer and KV head, the key/value rows those N CMEs produce in the frozen
  decoder (the Tier-1 K/V bank, gathered at the selected indices);
* the Tier-2 local window: a ring of W token slots per (sequence, layer,
  KV head), filled with W0 tokens before decoding starts (Section 2.5,
  "Tier-2: local context window" and "KV cache assembly");
* T decode steps, each appending one token to the ring and attending over
  [Tier-1 | Tier-2] with Hq query heads grouped over Hkv KV heads.

Inputs are Gaussian with the standard deviations below.  The shapes follow the
decoders the paper evaluates (Llama-3-8B-Instruct, Mistral-7B-Instruct-v0.3:
32 query heads, 8 KV heads, head_dim 128, hidden size 4096) and its cache
budgets (K in {30, 40}, W in {130, 256}, batch 8, up to 3,000 generated tokens;
hyperparameter table in the appendix), scaled up to the sizes of a serving
deployment.  They stand in for the SQuAD-based efficiency runs, whose data and
trained weights are not used here.
"""

from __future__ import annotations

import math
from dataclasses import dataclass, replace
from typing import Optional, Tuple


@dataclass(frozen=True)
class Workload:
    name: str
    B: int  # batch (independent sequences)
    L: int  # decoder layers in one decode step
    Hq: int  # query heads
    Hkv: int  # KV heads (GQA groups); Hq % Hkv == 0
    d: int  # head dimension
    N: int  # CMEs per sequence (the paper's M_b)
    D: int  # CME / question-vector dimension (the paper's H_d)
    k: int  # Tier-1 top-K
    W: int  # Tier-2 ring capacity (window length)
    T: int  # decode steps
    seed: int
    emb_std: float  # std of question-vector and CME entries
    kv_std: float  # std of K/V entries (Tier-1 bank, ring, appended tokens)
    q_std: float  # std of decode-query entries
    W0: Optional[Tuple[int, ...]] = None  # ring fill per sequence before step 0 (None: full)
    margin: float = 2e-4  # planted cosine gap at the top-k cut (0 disables planting)

    @property
    def G(self) -> int:
        return self.Hq // self.Hkv

    def fill(self) -> Tuple[int, ...]:
        """Tokens in each sequence's ring before the first decode step."""
        if self.W0 is None:
            return (self.W,) * self.B
        assert len(self.W0) == self.B
        return tuple(self.W0)

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


def _scaled(dim: int) -> float:
    return 1.0 / math.sqrt(dim)


# The five configurations.  "tiny" is the small case the oracle finishes in
# seconds; "llama3_8b" is the single-GPU throughput workload.
WORKLOADS = {
    "tiny": Workload(
        name="tiny", B=1, L=1, Hq=8, Hkv=2, d=64, N=256, D=512, k=32, W=128, T=16,
        seed=0, emb_std=_scaled(512), kv_std=1.0, q_std=_scaled(64),
    ),
    "llama3_8b": Workload(
        name="llama3_8b", B=1, L=32, Hq=32, Hkv=8, d=128, N=1024, D=4096, k=128, W=512,
        T=3000, seed=1, emb_std=_scaled(4096), kv_std=_scaled(128), q_std=_scaled(128),
    ),
    # Single attention layer: the configuration names no layer count.
    "mistral_batched": Workload(
        name="mistral_batched", B=32, L=1, Hq=32, Hkv=8, d=128, N=2048, D=4096, k=256,
        W=1024, T=3000, seed=2, emb_std=_scaled(4096), kv_std=_scaled(128),
        q_std=_scaled(128),
    ),
    "long_context": Workload(
        name="long_context", B=8, L=1, Hq=32, Hkv=8, d=128, N=16384, D=4096, k=2048,
        W=2048, T=512, seed=3, emb_std=_scaled(4096), kv_std=_scaled(128),
        q_std=_scaled(128),
    ),
}

ABLATION_K = (0, 64, 256, 1024, "all")
ABLATION_W = (128, 512, 2048)
ABLATION_B = (1, 16, 64)


def ablation_workload(k, W: int, B: int, L: int = 1, T: int = 4) -> Workload:
    """One point of the Llama-3-8B-shaped ablation sweep (bank of 1,024 CMEs)."""
    N = 1024
    kk = N if k == "all" else int(k)
    return Workload(
        name=f"ablation_k{k}_W{W}_B{B}", B=B, L=L, Hq=32, Hkv=8, d=128, N=N, D=4096,
        k=kk, W=W, T=T, seed=4, emb_std=_scaled(4096), kv_std=_scaled(128),
        q_std=_scaled(128),
    )


def ablation_workloads(L: int = 1, T: int = 4):
    return [ablation_workload(k, W, B, L=L, T=T)
            for k in ABLATION_K for W in ABLATION_W for B in ABLATION_B]


def full_window_workload(B: int = 1, T: int = 8) -> Workload:
    """k = all CMEs and a window that never evicts: the two-tier cache then holds
    every token, which is the equivalence case against plain attention."""
    W0 = 512
    return Workload(
        name="ablation_kall_Wfull", B=B, L=1, Hq=32, Hkv=8, d=128, N=1024, D=4096,
        k=1024, W=W0 + T, T=T, seed=4, emb_std=_scaled(4096), kv_std=_scaled(128),
        q_std=_scaled(128), W0=(W0,) * B,
    )


def get_workload(name: str) -> Workload:
    return WORKLOADS[name]
