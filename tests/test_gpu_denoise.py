"""Graph-based context denoising on the GPU against the fp64 oracle, stage
by stage.  The threshold test compares a cosine with tau in fp32 on both
sides; fp32 accumulation at H = 1280 is good to ~1e-6, and a long context
has cosines closer than that to any tau.  So: every token's pass flag (left
in the workspace) must equal the oracle's wherever no cosine of that token
lies within 2e-5 of tau, and the kept positions must equal, exactly, the
oracle's keep-minimum applied to the GPU's own pass flags.  Small cases also
compare the whole result with the oracle."""

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
import paper_2609_25537_gb300 as cmc
from workloads import WORKLOADS, context_inputs

pytestmark = pytest.mark.gpu

MARGIN = 2e-5


def _ambiguous(emb_b, n, g, tau):
    """Tokens whose test involves a cosine within MARGIN of tau."""
    amb = np.zeros(n, dtype=bool)
    e = torch.from_numpy(emb_b[:n]).double()
    for s in range(1, g + 1):
        if n > s:
            c = F.cosine_similarity(e[:-s], e[s:], dim=1, eps=0.0).numpy()
            amb[:-s] |= np.abs(c - tau) <= MARGIN
    return amb


def _check(emb, n_tok, g, tau, every, dev, pass_n_tokens=True, whole=True, ws=None):
    B, n_max, _ = emb.shape
    if ws is None:
        ws = torch.zeros(cmc.lib().cmc_denoise_workspace_size(B, n_max), dtype=torch.uint8,
                         device=dev)
    kept, cnt = cmc.denoise(torch.from_numpy(emb).to(dev),
                            n_tokens=torch.from_numpy(n_tok).to(dev) if pass_n_tokens else None,
                            g=g, tau=tau, keep_every=every, workspace=ws)
    torch.cuda.synchronize()
    kept, cnt = kept.cpu().numpy(), cnt.cpu().numpy()
    flags = ws[:B * n_max].cpu().numpy().reshape(B, n_max).astype(bool)
    for b in range(B):
        n = int(n_tok[b])
        want = oracle.denoise_pass(emb[b], n, g, tau)
        amb = _ambiguous(emb[b], n, g, tau)
        np.testing.assert_array_equal(flags[b, :n][~amb], want[~amb])
        assert not flags[b, n:].any()
        k = np.flatnonzero(oracle.keep_minimum(flags[b, :n], every))
        assert cnt[b] == k.size
        np.testing.assert_array_equal(kept[b, :k.size], k)
        assert np.all(kept[b, k.size:] == -1)
    if whole:
        ridx, rcnt = oracle.denoise(emb, n_tok, g, tau, every)
        np.testing.assert_array_equal(cnt, rcnt)
        np.testing.assert_array_equal(kept, ridx)
    return cnt


@pytest.mark.parametrize("name,H,ratio,batch", [
    ("tiny", 256, 4, None), ("llama3_8b", 1280, 4, None), ("long_context", 1280, 8, range(0, 1)),
])
def test_denoise_workloads(cuda_device, name, H, ratio, batch):
    w = WORKLOADS[name] if name != "tiny" else WORKLOADS["tiny"].with_(B=3)
    ci = context_inputs(w, H=H, ratio=ratio, batch=batch)
    cnt = _check(ci.emb, ci.n_tokens, 3, 0.05, 16, cuda_device, whole=name == "tiny")
    assert np.all(cnt >= ci.n_tokens // 16)          # the keep-minimum floor


def test_denoise_edge_cases(cuda_device):
    """g = 1 and g = 8, no keep-minimum, tau below -1 (all but the last token)
    and above 1 (only the keep-minimum), padding rows that must not be read
    (NaN), an empty and a one-token context, and no n_tokens (all rows)."""
    rng = np.random.default_rng(21)
    B, n, H = 4, 300, 64
    steps = rng.standard_normal((B, n, H)).astype(np.float32)
    emb = np.cumsum(steps, axis=1).astype(np.float32)
    n_tok = np.array([300, 217, 0, 1], dtype=np.int32)
    for b in range(B):
        emb[b, n_tok[b]:] = np.nan
    for g, every in ((1, 16), (8, 16), (3, 0), (3, 5)):
        _check(emb, n_tok, g, 0.3, every, cuda_device)
    cnt = _check(emb, n_tok, 3, -2.0, 16, cuda_device)
    assert cnt.tolist() == [299, 216, 0, 0]
    cnt = _check(emb, n_tok, 3, 2.0, 16, cuda_device)
    assert cnt.tolist() == [300 // 16, 217 // 16, 0, 0]
    full = np.nan_to_num(emb, nan=1.0)
    _check(full, np.full(B, n, dtype=np.int32), 3, 0.3, 16, cuda_device, pass_n_tokens=False)


def test_denoise_one_launch_and_two_launch_paths(cuda_device):
    """Contexts of 256 tiles of 32 tokens (the compaction runs in the pass
    launch, counted per context in the workspace) and of 257 (the cluster
    compaction kernel), one and several contexts, ragged last tiles; the same
    workspace serves repeated calls and its counters are zero after each."""
    rng = np.random.default_rng(5)
    H = 128
    for B, tiles in ((1, 256), (1, 257), (3, 256), (2, 3)):
        n_max = 32 * tiles - 7                     # a ragged last tile
        steps = rng.standard_normal((B, n_max, H)).astype(np.float32)
        emb = np.cumsum(steps, axis=1).astype(np.float32)
        n_tok = np.array([n_max - 45 * b for b in range(B)], dtype=np.int32)
        ws = torch.zeros(cmc.lib().cmc_denoise_workspace_size(B, n_max), dtype=torch.uint8,
                         device=cuda_device)
        for rep in range(3):
            _check(emb, n_tok, 3, 0.3, 16, cuda_device, whole=rep == 0, ws=ws)
            tail = ws[-256:].cpu().numpy()
            assert not tail.any(), "completion counters not left at zero"
