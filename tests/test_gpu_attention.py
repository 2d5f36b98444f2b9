"""Two-tier decode attention (and the ring append) on the GPU against the fp64
oracle, on the seeded workloads and on edge cases.

Full-size workloads run every decode step on the GPU and compare every head
of every layer at sampled steps (first steps, around the ring's wrap, middle,
last), with the oracle replaying the same appends.

Both Tier-1 forms are covered: "gather" passes the per-CME bank and idx to
every step; "dense" compacts the selected rows once with tier1_gather and
passes idx=None.  The oracle always gathers from the bank itself."""

import numpy as np
import pytest
import torch

import oracle
import paper_2609_25537_gb300 as cmc
from workloads import (WORKLOADS, kv_inputs, random_tier1_indices, selection_inputs,
                       step_inputs)
from workloads.configs import ablation_workloads, full_window_workload
from _gpu_helpers import assert_attn_close, dev_bf16, host_bits, to_f64

pytestmark = pytest.mark.gpu


MODES = ["gather", "dense"]


class Problem:
    """Device and host (oracle) copies of one decode problem.

    mode "gather": the attention calls get the bank and idx; "dense": the
    selected rows are compacted once by tier1_gather (checked bit-exact
    against indexing the host bank) and the calls get idx=None."""

    def __init__(self, w, dev, idx=None, mode="gather"):
        self.w = w
        self.dev = dev
        kv = kv_inputs(w)
        self.kv = kv
        if idx is None and w.k > 0:
            idx = random_tier1_indices(w)
        self.idx_host = None if w.k == 0 else np.asarray(idx, dtype=np.int64)
        self.idx = (torch.empty((w.B, 0), dtype=torch.int32, device=dev) if w.k == 0 else
                    torch.from_numpy(np.asarray(idx, dtype=np.int32)).to(dev))
        self.t1k, self.t1v = dev_bf16(kv.tier1_k, dev), dev_bf16(kv.tier1_v, dev)
        self.mode = mode if w.k > 0 else "gather"
        if self.mode == "dense":
            self.t1k, self.t1v = cmc.tier1_gather(self.t1k, self.t1v, self.idx)
            for dev_t, host in ((self.t1k, kv.tier1_k), (self.t1v, kv.tier1_v)):
                want = np.stack([host[b][:, :, self.idx_host[b]] for b in range(w.B)])
                np.testing.assert_array_equal(host_bits(dev_t), want)
            self.idx = None
        self.ring_k, self.ring_v = dev_bf16(kv.ring_k, dev), dev_bf16(kv.ring_v, dev)
        self.pos = torch.from_numpy(kv.pos0.copy()).to(dev)
        self.o_ring_k, self.o_ring_v = kv.ring_k.copy(), kv.ring_v.copy()
        self.o_pos = kv.pos0.copy()
        dims = cmc.dims_of(torch.empty(w.B, w.L, w.Hq, w.d, dtype=torch.bfloat16),
                           torch.empty(w.B, w.L, w.Hkv, w.N, w.d, dtype=torch.bfloat16),
                           self.idx, torch.empty(w.B, w.L, w.Hkv, w.W, w.d,
                                                 dtype=torch.bfloat16))
        self.ws = cmc.DecodeWorkspace(dims, dev)

    def step(self, st, q_dev=None, compare=True, scale=None):
        q_dev = dev_bf16(st.q, self.dev) if q_dev is None else q_dev
        out = cmc.decode_step(q_dev, self.t1k, self.t1v, self.idx, self.ring_k, self.ring_v,
                              self.pos, dev_bf16(st.k_new, self.dev),
                              dev_bf16(st.v_new, self.dev), workspace=self.ws, scale=scale)
        if not compare:
            oracle.window_append(self.o_ring_k, self.o_ring_v, self.o_pos, st.k_new, st.v_new)
            return out, None
        ref = oracle.decode_step(st.q, self.kv.tier1_k, self.kv.tier1_v, self.idx_host,
                                 self.o_ring_k, self.o_ring_v, self.o_pos, st.k_new, st.v_new,
                                 scale=scale)
        return out, ref

    def check_state(self):
        torch.cuda.synchronize()
        np.testing.assert_array_equal(self.pos.cpu().numpy(), self.o_pos)
        np.testing.assert_array_equal(host_bits(self.ring_k), self.o_ring_k)
        np.testing.assert_array_equal(host_bits(self.ring_v), self.o_ring_v)
        assert self.ws.status() == 0


@pytest.mark.parametrize("mode", MODES)
def test_tiny_every_step(cuda_device, mode):
    w = WORKLOADS["tiny"]
    si = selection_inputs(w)
    idx_ref, _ = oracle.score_select(si.question_emb, si.cme_bank, w.k)
    P = Problem(w, cuda_device, idx=idx_ref, mode=mode)
    for t in range(w.T):
        out, ref = P.step(step_inputs(w, t))
        assert_attn_close(to_f64(out), ref, f"tiny step {t}")
    P.check_state()


@pytest.mark.parametrize("q_scale", [3.0])
def test_tiny_peaked(cuda_device, q_scale):
    """Unscaled-style queries: logits with std ~3, so the softmax is peaked."""
    w = WORKLOADS["tiny"]
    P = Problem(w, cuda_device)
    for t in range(4):
        out, ref = P.step(step_inputs(w, t, q_std=q_scale / w.kv_std))
        assert_attn_close(to_f64(out), ref, f"tiny peaked step {t}")


def _sampled_run(w, dev, sample_steps, idx=None, q_std=None, mode="gather"):
    P = Problem(w, dev, idx=idx, mode=mode)
    q_fill = dev_bf16(step_inputs(w, 0, parts="q", q_std=q_std).q, dev)
    sample_steps = set(sample_steps)
    for t in range(w.T):
        if t in sample_steps:
            st = step_inputs(w, t, q_std=q_std)
            out, ref = P.step(st)
            assert_attn_close(to_f64(out), ref, f"{w.name} step {t}")
        else:
            st = step_inputs(w, t, parts="kv")
            P.step(st, q_dev=q_fill, compare=False)
    P.check_state()


def _samples(w):
    return sorted({0, 1, 2, w.W - 1, w.W, w.W + 1, w.T // 2, w.T - 1} & set(range(w.T)))


@pytest.mark.parametrize("mode", MODES)
def test_llama3_8b_full(cuda_device, mode):
    """The 32-layer Llama-3-8B-shaped workload, all 3,000 steps, with the
    selection taken from the Tier-1 scoring of its own CME bank."""
    w = WORKLOADS["llama3_8b"]
    si = selection_inputs(w)
    idx = cmc.score_select(torch.from_numpy(si.question_emb).to(cuda_device),
                           torch.from_numpy(si.cme_bank).to(cuda_device), w.k)
    idx_host = idx.cpu().numpy()
    np.testing.assert_array_equal(idx_host, oracle.score_select(si.question_emb, si.cme_bank,
                                                                w.k)[0])
    _sampled_run(w, cuda_device, _samples(w), idx=idx_host, mode=mode)


@pytest.mark.parametrize("mode", MODES)
def test_llama3_8b_peaked(cuda_device, mode):
    w = WORKLOADS["llama3_8b"].with_(T=3, L=4)
    _sampled_run(w, cuda_device, range(3), q_std=3.0 / w.kv_std, mode=mode)


@pytest.mark.parametrize("mode", MODES)
def test_mistral_batched_full(cuda_device, mode):
    w = WORKLOADS["mistral_batched"]
    _sampled_run(w, cuda_device, _samples(w), mode=mode)


@pytest.mark.parametrize("mode", MODES)
def test_long_context_full(cuda_device, mode):
    w = WORKLOADS["long_context"]
    _sampled_run(w, cuda_device, _samples(w), mode=mode)


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("w", ablation_workloads(L=1, T=3), ids=lambda w: w.name)
def test_ablation_grid(cuda_device, w, mode):
    _sampled_run(w, cuda_device, [0, w.T - 1], mode=mode)


@pytest.mark.parametrize("mode", MODES)
def test_all_cmes_unbounded_window_is_plain_attention(cuda_device, mode):
    """k = N and a window that never evicts: GPU output equals the oracle and
    plain softmax attention over [whole bank | every token so far]."""
    w = full_window_workload(B=2, T=6)
    P = Problem(w, cuda_device, idx=np.tile(np.arange(w.N), (w.B, 1)), mode=mode)
    hist_k = [list(P.kv.ring_k[b, :, :, :P.kv.pos0[b]].transpose(2, 0, 1, 3))
              for b in range(w.B)]
    hist_v = [list(P.kv.ring_v[b, :, :, :P.kv.pos0[b]].transpose(2, 0, 1, 3))
              for b in range(w.B)]
    for t in range(w.T):
        st = step_inputs(w, t)
        out, ref = P.step(st)
        got = to_f64(out)
        assert_attn_close(got, ref, f"full-window step {t}")
        for b in range(w.B):
            hist_k[b].append(st.k_new[b])
            hist_v[b].append(st.v_new[b])
        # plain attention for a few heads
        for b, l, h in [(0, 0, 0), (1, 0, 13), (1, 0, 31)]:
            g = h // w.G
            K = np.concatenate([oracle.bf16_to_f64(P.kv.tier1_k[b, l, g]),
                                oracle.bf16_to_f64(np.stack(hist_k[b])[:, l, g])])
            V = np.concatenate([oracle.bf16_to_f64(P.kv.tier1_v[b, l, g]),
                                oracle.bf16_to_f64(np.stack(hist_v[b])[:, l, g])])
            qv = oracle.bf16_to_f64(st.q[b, l, h])
            z = K @ qv / np.sqrt(w.d)
            p = np.exp(z - z.max())
            plain = p @ V / p.sum()
            np.testing.assert_allclose(ref[b, l, h], plain, rtol=1e-10, atol=1e-12)
            assert_attn_close(got[b, l, h], plain, "plain attention")


@pytest.mark.parametrize("mode", MODES)
def test_fused_step_equals_append_then_attend(cuda_device, mode):
    """The fused step and the two separate calls give bit-identical results."""
    for w in (WORKLOADS["tiny"], WORKLOADS["llama3_8b"].with_(L=2, T=3)):
        A = Problem(w, cuda_device, mode=mode)
        Bp = Problem(w, cuda_device, mode=mode)
        for t in range(3):
            st = step_inputs(w, t)
            q = dev_bf16(st.q, cuda_device)
            out_a = cmc.decode_step(q, A.t1k, A.t1v, A.idx, A.ring_k, A.ring_v, A.pos,
                                    dev_bf16(st.k_new, cuda_device),
                                    dev_bf16(st.v_new, cuda_device), workspace=A.ws)
            cmc.window_append(Bp.ring_k, Bp.ring_v, Bp.pos, dev_bf16(st.k_new, cuda_device),
                              dev_bf16(st.v_new, cuda_device))
            out_b = cmc.two_tier_decode_attn(q, Bp.t1k, Bp.t1v, Bp.idx, Bp.ring_k, Bp.ring_v,
                                             Bp.pos, workspace=Bp.ws)
            torch.cuda.synchronize()
            assert torch.equal(out_a.view(torch.int16), out_b.view(torch.int16))
            assert torch.equal(A.ring_k, Bp.ring_k) and torch.equal(A.pos, Bp.pos)


@pytest.mark.parametrize("mode", MODES)
def test_deterministic(cuda_device, mode):
    w = WORKLOADS["llama3_8b"].with_(L=2)
    outs = []
    for _ in range(2):
        P = Problem(w, cuda_device, mode=mode)
        st = step_inputs(w, 0)
        out, _ = P.step(st, compare=False)
        outs.append(out.view(torch.int16).clone())
    assert torch.equal(outs[0], outs[1])


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("G,d", [(1, 64), (2, 128), (8, 64), (8, 128), (4, 64)])
def test_head_shapes(cuda_device, G, d, mode):
    Hkv = 2
    w = WORKLOADS["tiny"].with_(B=2, L=3, Hq=G * Hkv, Hkv=Hkv, d=d, N=70, k=9, W=33, T=4,
                                kv_std=1.0, q_std=1.0 / np.sqrt(d), W0=(33, 5))
    P = Problem(w, cuda_device, mode=mode)
    for t in range(w.T):
        out, ref = P.step(step_inputs(w, t))
        assert_attn_close(to_f64(out), ref, f"G={G} d={d} step {t}")
    P.check_state()


@pytest.mark.parametrize("mode", MODES)
def test_ragged_fill_and_wrap(cuda_device, mode):
    """Sequences at different ring fills, including empty, crossing the wrap."""
    w = WORKLOADS["tiny"].with_(B=5, W=16, k=7, T=20, W0=(0, 1, 9, 15, 16))
    P = Problem(w, cuda_device, mode=mode)
    for t in range(w.T):
        out, ref = P.step(step_inputs(w, t))
        assert_attn_close(to_f64(out), ref, f"ragged step {t}")
    P.check_state()


@pytest.mark.parametrize("mode", MODES)
def test_window_of_one(cuda_device, mode):
    w = WORKLOADS["tiny"].with_(W=1, k=3, T=5)
    P = Problem(w, cuda_device, mode=mode)
    for t in range(w.T):
        out, ref = P.step(step_inputs(w, t))
        assert_attn_close(to_f64(out), ref, f"W=1 step {t}")
    P.check_state()


def test_k_zero_and_empty_cache(cuda_device):
    w = WORKLOADS["tiny"].with_(k=0, B=2, W0=(0, 40), T=3)
    P = Problem(w, cuda_device)
    # attention without append on an empty ring: zero output for sequence 0
    st = step_inputs(w, 0)
    out = cmc.two_tier_decode_attn(dev_bf16(st.q, cuda_device), P.t1k, P.t1v, P.idx, P.ring_k,
                                   P.ring_v, P.pos, workspace=P.ws)
    ref = oracle.two_tier_attention(st.q, P.kv.tier1_k, P.kv.tier1_v, None, P.o_ring_k,
                                    P.o_ring_v, P.o_pos)
    got = to_f64(out)
    assert np.all(got[0] == 0.0)
    assert_attn_close(got, ref, "k=0 attention-only")
    for t in range(w.T):
        out, ref = P.step(step_inputs(w, t))
        assert_attn_close(to_f64(out), ref, f"k=0 step {t}")
    P.check_state()


@pytest.mark.parametrize("mode", MODES)
def test_unsorted_idx_and_explicit_scale(cuda_device, mode):
    w = WORKLOADS["tiny"].with_(T=2)
    idx = random_tier1_indices(w)
    perm = np.random.default_rng(0).permutation(w.k)
    P = Problem(w, cuda_device, idx=idx[:, perm], mode=mode)
    for t in range(w.T):
        out, ref = P.step(step_inputs(w, t), scale=0.05)
        assert_attn_close(to_f64(out), ref, f"unsorted idx step {t}")


def test_bad_index_and_bad_pos_are_flagged_and_skipped(cuda_device):
    w = WORKLOADS["tiny"].with_(B=3, T=1)
    idx = random_tier1_indices(w).astype(np.int64)
    idx[1, 3] = -1
    idx[1, 10] = w.N
    P = Problem(w, cuda_device, idx=idx)
    P.pos[2] = -5
    st = step_inputs(w, 0)
    out = cmc.decode_step(dev_bf16(st.q, cuda_device), P.t1k, P.t1v, P.idx, P.ring_k, P.ring_v,
                          P.pos, dev_bf16(st.k_new, cuda_device),
                          dev_bf16(st.v_new, cuda_device), workspace=P.ws)
    flags = P.ws.status()
    assert flags == cmc.DEVFLAG_BAD_INDEX | cmc.DEVFLAG_BAD_POS
    got = to_f64(out)
    # sequence 2: zero output, ring and pos untouched
    assert np.all(got[2] == 0.0)
    assert int(P.pos[2]) == -5
    np.testing.assert_array_equal(host_bits(P.ring_k)[2], P.kv.ring_k[2])
    # sequences 0 and 1: the oracle with the bad rows removed
    keep = [np.array([i for i in row if 0 <= i < w.N]) for row in idx[:2]]
    ring_k, ring_v = P.kv.ring_k[:2].copy(), P.kv.ring_v[:2].copy()
    pos = P.kv.pos0[:2].copy()
    oracle.window_append(ring_k, ring_v, pos, st.k_new[:2], st.v_new[:2])
    for b in range(2):
        for h in range(w.Hq):
            ref = oracle.two_tier_attention_head(st.q, P.kv.tier1_k, P.kv.tier1_v,
                                                 {b: keep[b]}, ring_k, ring_v, pos, b, 0, h)
            assert_attn_close(got[b, 0, h], ref, f"bad idx b={b} h={h}")


@pytest.mark.parametrize("mode", MODES)
def test_large_unit_count(cuda_device, mode):
    """B * L * Hkv = 16,384 units in one launch (batch 64, 32 layers)."""
    w = WORKLOADS["llama3_8b"].with_(B=64, L=32, N=40, k=8, W=24, T=1, W0=None)
    P = Problem(w, cuda_device, mode=mode)
    st = step_inputs(w, 0)
    out, _ = P.step(st, compare=False)
    got = to_f64(out)
    rng = np.random.default_rng(0)
    ring_k, ring_v, pos = P.o_ring_k, P.o_ring_v, P.o_pos
    for _ in range(64):
        b, l, h = int(rng.integers(w.B)), int(rng.integers(w.L)), int(rng.integers(w.Hq))
        ref = oracle.two_tier_attention_head(st.q, P.kv.tier1_k, P.kv.tier1_v, P.idx_host,
                                             ring_k, ring_v, pos, b, l, h)
        assert_attn_close(got[b, l, h], ref, f"unit sample {(b, l, h)}")
    P.check_state()


@pytest.mark.parametrize("mode", MODES)
def test_unoccupied_slots_holding_nan_do_not_leak(cuda_device, mode):
    """Ring slots past the fill (and so outside the cache) hold NaN on the
    device: masked keys must not reach the output, whatever memory holds."""
    w = WORKLOADS["tiny"].with_(B=3, W=100, k=40, T=3, W0=(0, 37, 64))
    P = Problem(w, cuda_device, mode=mode)
    nan = torch.tensor(0x7FC0, dtype=torch.int16).view(torch.bfloat16).to(cuda_device)
    for b, f in enumerate(w.fill()):
        P.ring_k[b, :, :, f:] = nan
        P.ring_v[b, :, :, f:] = nan
    for t in range(w.T):
        out, ref = P.step(step_inputs(w, t))
        got = to_f64(out)
        assert np.isfinite(got).all()
        assert_attn_close(got, ref, f"NaN-filled free slots step {t}")


def test_tier1_gather_bad_index_zero_row_and_flag(cuda_device):
    w = WORKLOADS["tiny"].with_(B=2, L=2)
    kv = kv_inputs(w)
    idx = random_tier1_indices(w).astype(np.int32)
    idx[1, 5] = w.N
    idx[0, 0] = -3
    dims = cmc.dims_of(torch.empty(w.B, w.L, w.Hq, w.d, dtype=torch.bfloat16),
                       torch.empty(w.B, w.L, w.Hkv, w.N, w.d, dtype=torch.bfloat16),
                       None, torch.empty(w.B, w.L, w.Hkv, w.W, w.d, dtype=torch.bfloat16))
    ws = cmc.DecodeWorkspace(dims, cuda_device)
    tk, tv = cmc.tier1_gather(dev_bf16(kv.tier1_k, cuda_device), dev_bf16(kv.tier1_v, cuda_device),
                              torch.from_numpy(idx).to(cuda_device), workspace=ws)
    assert ws.status() == cmc.DEVFLAG_BAD_INDEX
    for dev_t, host in ((tk, kv.tier1_k), (tv, kv.tier1_v)):
        got = host_bits(dev_t)
        for b in range(w.B):
            for i, j in enumerate(idx[b]):
                want = host[b][:, :, j] if 0 <= j < w.N else 0
                np.testing.assert_array_equal(got[b][:, :, i], want)


def test_decode_attn_plan(cuda_device):
    """One CTA per (layer, KV head) unit and a single launch per step at the
    Llama-3-8B shape when 256 CTAs fit in one wave; the long-context shape's
    long units are split over clusters, still one launch."""
    sms = torch.cuda.get_device_properties(cuda_device).multi_processor_count
    w = WORKLOADS["llama3_8b"]
    dims = cmc.CmcDims(w.B, w.L, w.Hq, w.Hkv, w.d, w.k, w.k, w.W)
    ctas, launches = cmc.decode_attn_plan(dims)
    if 2 * sms >= 256:
        assert (ctas, launches) == (256, 1)
    w = WORKLOADS["long_context"]
    dims = cmc.CmcDims(w.B, w.L, w.Hq, w.Hkv, w.d, w.k, w.k, w.W)
    ctas, launches = cmc.decode_attn_plan(dims, fused=False)
    assert launches in (1, 2) and ctas >= 64
    if 2 * sms >= 256:
        # 64 units of 64 tiles, four CTAs per unit: clusters merged in
        # distributed shared memory, no combine launch
        assert (ctas, launches) == (256, 1)


def _cluster_case(B, L, Hkv, k, W, N=None, T=3, G=4, d=128):
    return WORKLOADS["tiny"].with_(B=B, L=L, Hq=G * Hkv, Hkv=Hkv, d=d, N=N or max(k, 1) + 17, k=k,
                                   W=W, T=T, kv_std=1.0 / np.sqrt(d), q_std=1.0 / np.sqrt(d),
                                   W0=tuple((W * (i + 1)) // B for i in range(B)))


# (B, L, Hkv, k, W): units B*L*Hkv, tiles per unit ceil(k/64) + ceil(W/64);
# on 152 SMs with two CTAs each these give clusters of 2, 3, 5 and 8 CTAs per
# unit, the last capped at 8 (20 would fit)
CLUSTER_CASES = [(19, 1, 8, 64, 64), (1, 1, 2, 32, 128), (15, 1, 4, 128, 192),
                 (19, 2, 1, 256, 256), (1, 1, 2, 640, 640)]


@pytest.mark.parametrize("extra,launches", [(17, 2), (None, 1)])
def test_more_units_than_ctas(cuda_device, extra, launches):
    """More units than resident CTAs.  A few units over a multiple of the CTA
    count: tiles split evenly (units cut between CTAs) and the combine kernel
    merges them.  Half again as many: whole units per CTA, one launch.  Parity
    over ragged fills either way."""
    sms = torch.cuda.get_device_properties(cuda_device).multi_processor_count
    B = 2 * sms + extra if extra is not None else 3 * sms // 2
    w = _cluster_case(B, 1, 2, 64, 128, T=2)
    dims = cmc.CmcDims(w.B, w.L, w.Hq, w.Hkv, w.d, w.N, w.k, w.W)
    ctas, got = cmc.decode_attn_plan(dims)
    two_per_sm = cmc.decode_attn_plan(cmc.CmcDims(2 * sms + 1, 1, 4, 1, 128, 64, 64, 64))[0] == 2 * sms
    if two_per_sm:
        assert (ctas, got) == (2 * sms, launches)
    P = Problem(w, cuda_device, mode="dense")
    for t in range(w.T):
        out, ref = P.step(step_inputs(w, t))
        assert_attn_close(to_f64(out), ref, f"{w.B * w.Hkv} units step {t}")
    P.check_state()


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("case", CLUSTER_CASES, ids=lambda c: "x".join(map(str, c)))
def test_split_units(cuda_device, case, mode):
    """Units shared by several CTAs: each plan's launches, and parity with
    the oracle over ragged fills (some CTAs of a unit hold no key)."""
    B, L, Hkv, k, W = case
    w = _cluster_case(B, L, Hkv, k, W)
    tpu = -(-k // 64) + -(-W // 64)
    units = B * L * Hkv
    sms = torch.cuda.get_device_properties(cuda_device).multi_processor_count
    dims = cmc.CmcDims(w.B, w.L, w.Hq, w.Hkv, w.d, w.N, w.k, w.W)
    ctas, launches = cmc.decode_attn_plan(dims)
    m = min((2 * sms) // units, tpu, 8)
    # two resident CTAs per SM (the plan of more units than that fills them)
    two_per_sm = cmc.decode_attn_plan(cmc.CmcDims(2 * sms + 1, 1, 4, 1, 128, 64, 64, 64))[0] == 2 * sms
    if two_per_sm and 2 * sms >= units:
        assert ctas == units * m
        assert launches == 1
    P = Problem(w, cuda_device, mode=mode)
    for t in range(w.T):
        out, ref = P.step(step_inputs(w, t))
        assert_attn_close(to_f64(out), ref, f"split units {case} step {t}")
    P.check_state()


@pytest.mark.parametrize("G,d", [(8, 128), (1, 64), (2, 64), (8, 64)])
def test_split_units_head_shapes(cuda_device, G, d):
    """Clusters of 3 and 5 CTAs per unit with other query-group sizes and head
    dimensions (the merge's share of output columns per CTA differs)."""
    for case in ((1, 1, 2, 32, 128), (15, 1, 4, 128, 192)):
        w = _cluster_case(*case, G=G, d=d)
        P = Problem(w, cuda_device, mode="dense")
        for t in range(w.T):
            out, ref = P.step(step_inputs(w, t))
            assert_attn_close(to_f64(out), ref, f"split units {case} G={G} d={d} step {t}")
        P.check_state()


# ----------------------------------------------------------------------------
# Decode step of a GQA layer with rotary position embedding
# ----------------------------------------------------------------------------

def _ring_close_bf16(got_bits, want_bits, what, max_frac=2e-3):
    """Rotated keys are rounded to bf16 on both sides, from fp32 (GPU) and fp64
    (oracle) values.  They may round to neighbouring bf16 values (one unit in
    the last place: 2^-7 relative), and where the rotation cancels to almost 0
    the fp32 error (~1e-7 of the inputs) shows; both rarely."""
    a = oracle.bf16_to_f64(got_bits)
    b = oracle.bf16_to_f64(want_bits)
    err = np.abs(a - b)
    bound = 2.0 ** -7 * np.abs(b) + 1e-6 * np.abs(b).max()
    assert np.all(err <= bound), f"{what}: max excess {(err - bound).max():.3e}"
    assert (err != 0).mean() <= max_frac, f"{what}: {(err != 0).mean():.2e} of elements differ"


def _rope_run(w, dev, mode, theta, offset, compare_steps=None, q_std=None):
    P = Problem(w, dev, mode=mode)
    steps = range(w.T) if compare_steps is None else compare_steps
    for t in range(w.T):
        st = step_inputs(w, t, q_std=q_std)
        out = cmc.decode_step(dev_bf16(st.q, dev), P.t1k, P.t1v, P.idx, P.ring_k, P.ring_v, P.pos,
                              dev_bf16(st.k_new, dev), dev_bf16(st.v_new, dev), workspace=P.ws,
                              rope_theta=theta, rope_offset=offset)
        ref = oracle.decode_step_rope(st.q, P.kv.tier1_k, P.kv.tier1_v, P.idx_host, P.o_ring_k,
                                      P.o_ring_v, P.o_pos, st.k_new, st.v_new, theta=theta,
                                      rope_offset=offset)
        if t in steps:
            assert_attn_close(to_f64(out), ref, f"{w.name} rope step {t}")
    torch.cuda.synchronize()
    np.testing.assert_array_equal(P.pos.cpu().numpy(), P.o_pos)
    np.testing.assert_array_equal(host_bits(P.ring_v), P.o_ring_v)
    _ring_close_bf16(host_bits(P.ring_k), P.o_ring_k, f"{w.name} rotated keys")
    assert P.ws.status() == 0


@pytest.mark.parametrize("mode", MODES)
def test_rope_tiny_every_step(cuda_device, mode):
    w = WORKLOADS["tiny"]
    _rope_run(w, cuda_device, mode, theta=10000.0, offset=w.k)


@pytest.mark.parametrize("mode", MODES)
def test_rope_llama_shape(cuda_device, mode):
    w = WORKLOADS["llama3_8b"].with_(L=4, T=6)
    _rope_run(w, cuda_device, mode, theta=500000.0, offset=w.k)


def test_rope_large_positions_and_peaked_queries(cuda_device):
    """Positions past 10^5 (long contexts): angles of 10^5 rad and more, which
    the kernel reduces to turns with 64-bit integer arithmetic."""
    w = WORKLOADS["tiny"].with_(B=2, T=4, kv_std=0.3)
    _rope_run(w, cuda_device, "dense", theta=10000.0, offset=123457, q_std=3.0 / 0.3)


@pytest.mark.parametrize("G,d", [(1, 64), (2, 128), (8, 64), (8, 128)])
def test_rope_head_shapes_ragged(cuda_device, G, d):
    Hkv = 2
    w = WORKLOADS["tiny"].with_(B=3, L=2, Hq=G * Hkv, Hkv=Hkv, d=d, N=70, k=9, W=33, T=5,
                                kv_std=1.0, q_std=1.0 / np.sqrt(d), W0=(33, 5, 0))
    _rope_run(w, cuda_device, "gather", theta=1e6, offset=w.k)


def test_rope_at_position_zero_equals_the_plain_step(cuda_device):
    """p = 0 rotates by nothing: the output and ring are bit-identical to the
    fused step without rotary embedding."""
    w = WORKLOADS["llama3_8b"].with_(L=2, T=1, B=2, W0=(0, 0))
    A = Problem(w, cuda_device, mode="dense")
    Bp = Problem(w, cuda_device, mode="dense")
    st = step_inputs(w, 0)
    args = lambda P: (dev_bf16(st.q, cuda_device), P.t1k, P.t1v, P.idx, P.ring_k, P.ring_v, P.pos,
                      dev_bf16(st.k_new, cuda_device), dev_bf16(st.v_new, cuda_device))
    out_a = cmc.decode_step(*args(A), workspace=A.ws)
    out_b = cmc.decode_step(*args(Bp), workspace=Bp.ws, rope_theta=500000.0, rope_offset=0)
    torch.cuda.synchronize()
    assert torch.equal(out_a.view(torch.int16), out_b.view(torch.int16))
    assert torch.equal(A.ring_k, Bp.ring_k) and torch.equal(A.pos, Bp.pos)


def test_rope_plan_matches_the_fused_step(cuda_device):
    w = WORKLOADS["llama3_8b"]
    dims = cmc.CmcDims(w.B, w.L, w.Hq, w.Hkv, w.d, w.k, w.k, w.W)
    assert cmc.decode_attn_plan(dims, rope=True) == cmc.decode_attn_plan(dims)


def _rope_append_host(P, st, theta, offset):
    """The oracle side of a step whose output is not compared: the new key
    rotated at its position and rounded to bf16, then appended with the value
    (the first half of oracle.decode_step_rope)."""
    k_rot = np.empty(st.k_new.shape, dtype=np.uint16)
    for b in range(P.w.B):
        p = offset + int(P.o_pos[b])
        k_rot[b] = oracle.f64_to_bf16_bits(oracle.rope_rotate(st.k_new[b], p, theta))
    oracle.window_append(P.o_ring_k, P.o_ring_v, P.o_pos, k_rot, st.v_new)


def _rope_sampled_run(w, dev, mode, theta, offset, sample_steps):
    """Every step runs the rotary decode step on the GPU; the outputs of the
    sampled steps are compared with oracle.decode_step_rope, and the ring and
    pos after the last step with the oracle's replay of every append."""
    P = Problem(w, dev, mode=mode)
    sample_steps = set(sample_steps)
    q_fill = dev_bf16(step_inputs(w, 0, parts="q").q, dev)
    for t in range(w.T):
        if t in sample_steps:
            st = step_inputs(w, t)
            q_dev = dev_bf16(st.q, dev)
        else:
            st = step_inputs(w, t, parts="kv")
            q_dev = q_fill
        out = cmc.decode_step(q_dev, P.t1k, P.t1v, P.idx, P.ring_k, P.ring_v, P.pos,
                              dev_bf16(st.k_new, dev), dev_bf16(st.v_new, dev), workspace=P.ws,
                              rope_theta=theta, rope_offset=offset)
        if t in sample_steps:
            ref = oracle.decode_step_rope(st.q, P.kv.tier1_k, P.kv.tier1_v, P.idx_host,
                                          P.o_ring_k, P.o_ring_v, P.o_pos, st.k_new, st.v_new,
                                          theta=theta, rope_offset=offset)
            assert_attn_close(to_f64(out), ref, f"{w.name} rope step {t}")
        else:
            _rope_append_host(P, st, theta, offset)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(P.pos.cpu().numpy(), P.o_pos)
    np.testing.assert_array_equal(host_bits(P.ring_v), P.o_ring_v)
    _ring_close_bf16(host_bits(P.ring_k), P.o_ring_k, f"{w.name} rotated keys")
    assert P.ws.status() == 0


def _two_ctas_per_sm(sms):
    return cmc.decode_attn_plan(cmc.CmcDims(2 * sms + 1, 1, 4, 1, 128, 64, 64, 64),
                                rope=True)[0] == 2 * sms


@pytest.mark.parametrize("mode", MODES)
def test_rope_llama_full_shape_one_cta_per_unit(cuda_device, mode):
    """The rotary step at the benchmarked shape: 32 layers, 256 units, one CTA
    per unit (the plan the bench times), Llama-3's theta = 5e5, through the
    ring's wrap: W + 2 steps, outputs compared at 0, 1, 2, W-1, W, W+1."""
    w = WORKLOADS["llama3_8b"]
    w = w.with_(T=w.W + 2)
    sms = torch.cuda.get_device_properties(cuda_device).multi_processor_count
    dims = cmc.CmcDims(w.B, w.L, w.Hq, w.Hkv, w.d, w.k, w.k, w.W)
    if _two_ctas_per_sm(sms) and 2 * sms >= 256:
        assert cmc.decode_attn_plan(dims, rope=True) == (256, 1)
    _rope_sampled_run(w, cuda_device, mode, theta=500000.0, offset=w.k,
                      sample_steps=[0, 1, 2, w.W - 1, w.W, w.W + 1])


def test_rope_whole_units_per_cta_several_sequences(cuda_device):
    """More units than resident CTAs, whole units per CTA: with one KV head per
    sequence, a CTA that takes two units takes two sequences, so the producer
    forms the rotary table of a second position inside one CTA's run."""
    sms = torch.cuda.get_device_properties(cuda_device).multi_processor_count
    B = 3 * sms
    w = _cluster_case(B, 1, 1, 64, 128, T=3)
    w = w.with_(W0=tuple((17 * b) % (w.W + 1) for b in range(B)))
    dims = cmc.CmcDims(w.B, w.L, w.Hq, w.Hkv, w.d, w.N, w.k, w.W)
    ctas, launches = cmc.decode_attn_plan(dims, rope=True)
    if _two_ctas_per_sm(sms):
        # 3 sms units on 2 sms CTAs: half of the CTAs take two whole units
        assert (ctas, launches) == (2 * sms, 1)
    P = Problem(w, cuda_device, mode="dense")
    for t in range(w.T):
        st = step_inputs(w, t)
        out = cmc.decode_step(dev_bf16(st.q, cuda_device), P.t1k, P.t1v, P.idx, P.ring_k,
                              P.ring_v, P.pos, dev_bf16(st.k_new, cuda_device),
                              dev_bf16(st.v_new, cuda_device), workspace=P.ws,
                              rope_theta=500000.0, rope_offset=w.k)
        ref = oracle.decode_step_rope(st.q, P.kv.tier1_k, P.kv.tier1_v, P.idx_host, P.o_ring_k,
                                      P.o_ring_v, P.o_pos, st.k_new, st.v_new, theta=500000.0,
                                      rope_offset=w.k)
        assert_attn_close(to_f64(out), ref, f"whole units rope step {t}")
    torch.cuda.synchronize()
    np.testing.assert_array_equal(P.pos.cpu().numpy(), P.o_pos)
    np.testing.assert_array_equal(host_bits(P.ring_v), P.o_ring_v)
    _ring_close_bf16(host_bits(P.ring_k), P.o_ring_k, "whole units rotated keys")
    assert P.ws.status() == 0


@pytest.mark.parametrize("mode", MODES)
def test_rope_stream_k_and_combine(cuda_device, mode):
    """A few units over a multiple of the CTA count: the tiles are split evenly
    (units cut between CTAs, runs of several sequences per CTA) and the combine
    kernel merges the cut units -- the rotary step on that plan."""
    sms = torch.cuda.get_device_properties(cuda_device).multi_processor_count
    B = 2 * sms + 17
    w = _cluster_case(B, 1, 2, 64, 128, T=3)
    dims = cmc.CmcDims(w.B, w.L, w.Hq, w.Hkv, w.d, w.N, w.k, w.W)
    ctas, launches = cmc.decode_attn_plan(dims, rope=True)
    if _two_ctas_per_sm(sms):
        assert (ctas, launches) == (2 * sms, 2)
    P = Problem(w, cuda_device, mode=mode)
    theta, offset = 500000.0, 3 * w.k + 5
    for t in range(w.T):
        st = step_inputs(w, t)
        out = cmc.decode_step(dev_bf16(st.q, cuda_device), P.t1k, P.t1v, P.idx, P.ring_k,
                              P.ring_v, P.pos, dev_bf16(st.k_new, cuda_device),
                              dev_bf16(st.v_new, cuda_device), workspace=P.ws,
                              rope_theta=theta, rope_offset=offset)
        ref = oracle.decode_step_rope(st.q, P.kv.tier1_k, P.kv.tier1_v, P.idx_host, P.o_ring_k,
                                      P.o_ring_v, P.o_pos, st.k_new, st.v_new, theta=theta,
                                      rope_offset=offset)
        assert_attn_close(to_f64(out), ref, f"stream-K rope step {t}")
    torch.cuda.synchronize()
    np.testing.assert_array_equal(P.pos.cpu().numpy(), P.o_pos)
    np.testing.assert_array_equal(host_bits(P.ring_v), P.o_ring_v)
    _ring_close_bf16(host_bits(P.ring_k), P.o_ring_k, "stream-K rotated keys")
    assert P.ws.status() == 0


def test_rope_frequency_table_in_device_memory_or_parameters(cuda_device):
    """The rotary frequencies come from a device table written on a theta's
    first use outside graph capture, or from the kernel parameters when that
    first use is being captured: both give bit-identical steps."""
    w = WORKLOADS["tiny"].with_(B=2, T=1)
    theta = 23456.789  # used by no other test
    A = Problem(w, cuda_device, mode="dense")
    Bp = Problem(w, cuda_device, mode="dense")
    st = step_inputs(w, 0)
    q, kn, vn = (dev_bf16(x, cuda_device) for x in (st.q, st.k_new, st.v_new))
    out_a = torch.empty_like(q)
    stream = torch.cuda.Stream(device=cuda_device)
    stream.wait_stream(torch.cuda.current_stream(cuda_device))
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        cmc.decode_step(q, A.t1k, A.t1v, A.idx, A.ring_k, A.ring_v, A.pos, kn, vn, out=out_a,
                        workspace=A.ws, rope_theta=theta, rope_offset=w.k)
    g.replay()
    torch.cuda.synchronize()
    out_b = cmc.decode_step(q, Bp.t1k, Bp.t1v, Bp.idx, Bp.ring_k, Bp.ring_v, Bp.pos, kn, vn,
                            workspace=Bp.ws, rope_theta=theta, rope_offset=w.k)
    torch.cuda.synchronize()
    assert torch.equal(out_a.view(torch.int16), out_b.view(torch.int16))
    assert torch.equal(A.ring_k, Bp.ring_k) and torch.equal(A.pos, Bp.pos)
    ref = oracle.decode_step_rope(st.q, A.kv.tier1_k, A.kv.tier1_v, A.idx_host, A.o_ring_k,
                                  A.o_ring_v, A.o_pos, st.k_new, st.v_new, theta=theta,
                                  rope_offset=w.k)
    assert_attn_close(to_f64(out_b), ref, "rope table paths")


def test_rope_many_thetas(cuda_device):
    """More distinct thetas than device table slots: the later ones use the
    kernel parameters; every step matches the oracle."""
    w = WORKLOADS["tiny"].with_(B=1, T=1)
    for j in range(20):
        _rope_run(w, cuda_device, "dense", theta=1000.0 + 97.5 * j, offset=w.k)


@pytest.mark.parametrize("tiles", [0, 64])
def test_l2_prefetch_depth_changes_no_result(cuda_device, tiles):
    """The pre-wait L2 prefetch depth is a hint: at the 32-layer Llama shape
    (dense Tier-1, one CTA per unit) steps with no prefetch or the deepest
    one give the same bits as the default depth of 5, and match the oracle."""
    w = WORKLOADS["llama3_8b"]
    idx = random_tier1_indices(w)
    outs = {}
    try:
        for depth in (5, tiles):
            cmc.set_l2_prefetch_tiles(depth)
            P = Problem(w, cuda_device, idx=idx, mode="dense")
            got = []
            for t in range(3):
                out, ref = P.step(step_inputs(w, t))
                assert_attn_close(to_f64(out), ref, f"prefetch {depth} step {t}")
                got.append(host_bits(out))
            P.check_state()
            outs[depth] = got
    finally:
        cmc.set_l2_prefetch_tiles(5)
    for a, b in zip(outs[5], outs[tiles]):
        np.testing.assert_array_equal(a, b)
