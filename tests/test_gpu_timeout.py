"""The attention kernel's bounded waits, made to run out on purpose.

cmc_test_stall_attention_waits(1) makes every pipeline stage expect 16 bytes
more than its loads deliver, so that no stage's barrier phase ever completes
(a wait that nothing ends: no access leaves its buffer and nothing traps).
Each CTA's first wait then gives up after its 1 s limit, the CTA's other
waits end at once, the producer warp gives its issued loads 2 ms to land, and
the call reports CMC_DEVFLAG_TIMEOUT in the workspace's status word.

Checked: the call returns, the flag is raised, and the context stays usable
-- with the hook off and the ring, pos and workspace restored, the same step
matches the fp64 oracle.  Launch plans: clusters of CTAs per unit (tiny) and
one CTA per unit (the 32-layer Llama shape: dense Tier-1, the plain and the
rotary-embedding step)."""

import time

import numpy as np
import pytest
import torch

import oracle
import paper_2609_25537_gb300 as cmc
from paper_2609_25537_gb300._lib import DEVFLAG_TIMEOUT
from workloads import WORKLOADS, kv_inputs, random_tier1_indices, step_inputs
from _gpu_helpers import assert_attn_close, dev_bf16, to_f64

pytestmark = pytest.mark.gpu

ROPE_THETA = 500000.0


@pytest.mark.parametrize("name,dense,rope", [("tiny", False, False), ("llama3_8b", True, False),
                                             ("llama3_8b", True, True)])
def test_stalled_waits_time_out_and_context_survives(cuda_device, name, dense, rope):
    dev = cuda_device
    w = WORKLOADS[name]
    kv = kv_inputs(w)
    idx_host = np.asarray(random_tier1_indices(w), dtype=np.int64)
    idx = torch.from_numpy(idx_host.astype(np.int32)).to(dev)
    t1k, t1v = dev_bf16(kv.tier1_k, dev), dev_bf16(kv.tier1_v, dev)
    if dense:
        t1k, t1v = cmc.tier1_gather(t1k, t1v, idx)
        idx = None
    st = step_inputs(w, 0)
    q, k_new, v_new = dev_bf16(st.q, dev), dev_bf16(st.k_new, dev), dev_bf16(st.v_new, dev)

    def state():
        return (dev_bf16(kv.ring_k, dev), dev_bf16(kv.ring_v, dev),
                torch.from_numpy(kv.pos0.copy()).to(dev))

    def step(ring_k, ring_v, pos, ws):
        kw = dict(rope_theta=ROPE_THETA, rope_offset=w.k) if rope else {}
        return cmc.decode_step(q, t1k, t1v, idx, ring_k, ring_v, pos, k_new, v_new,
                               workspace=ws, **kw)

    ring_k, ring_v, pos = state()
    dims = cmc.dims_of(q, t1k, idx, ring_k)
    torch.cuda.synchronize(dev)

    # stalled: every CTA's first wait runs out
    ws = cmc.DecodeWorkspace(dims, dev)
    assert cmc.lib().cmc_test_stall_attention_waits(1) == 0
    try:
        t0 = time.perf_counter()
        step(ring_k, ring_v, pos, ws)
        flags = ws.status()  # synchronises with the call
        elapsed = time.perf_counter() - t0
    finally:
        assert cmc.lib().cmc_test_stall_attention_waits(0) == 0
    assert flags & DEVFLAG_TIMEOUT, f"status {flags:#x}: no timeout reported"
    assert 0.9 <= elapsed < 30.0, f"stalled call took {elapsed:.2f} s (limit 1 s a wait)"
    assert ws.status() == 0  # read with clear: the flag is gone

    # the context is usable: the same step on restored state is exact again
    ring_k, ring_v, pos = state()
    ws = cmc.DecodeWorkspace(dims, dev)
    out = step(ring_k, ring_v, pos, ws)
    o_ring_k, o_ring_v, o_pos = kv.ring_k.copy(), kv.ring_v.copy(), kv.pos0.copy()
    if rope:
        ref = oracle.decode_step_rope(st.q, kv.tier1_k, kv.tier1_v, idx_host, o_ring_k, o_ring_v,
                                      o_pos, st.k_new, st.v_new, ROPE_THETA, w.k)
    else:
        ref = oracle.decode_step(st.q, kv.tier1_k, kv.tier1_v, idx_host, o_ring_k, o_ring_v,
                                 o_pos, st.k_new, st.v_new)
    assert_attn_close(to_f64(out), ref, f"{name} after the stalled call")
    assert ws.status() == 0
    np.testing.assert_array_equal(pos.cpu().numpy(), o_pos)
