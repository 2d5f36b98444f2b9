"""The multi-core timing of the oracle (bench.py's CPU baseline and reference
arm) runs the unchanged oracle on slices of a decode problem.  Sequences and
layers are independent within a decode step, so the slices' results put side
by side must equal the whole step's: checked here in one process, on both
slicing axes, with the ring state carried across steps."""

import numpy as np

import oracle
from oracle.host_pool import _slices, slice_problem
from workloads import WORKLOADS, kv_inputs, random_tier1_indices, step_inputs


def test_slices_cover_the_axis_once():
    for B, L, workers in [(1, 32, 16), (1, 32, 72), (32, 1, 16), (8, 4, 3), (5, 1, 8)]:
        axis, ranges = _slices(B, L, workers)
        n = B if axis == "b" else L
        assert len(ranges) == min(workers, n)
        assert ranges[0][0] == 0 and ranges[-1][1] == n
        assert all(a < b for a, b in ranges)
        assert all(ranges[i][1] == ranges[i + 1][0] for i in range(len(ranges) - 1))


def _check(w, workers):
    kv = kv_inputs(w)
    idx = random_tier1_indices(w).astype(np.int64)
    sts = [step_inputs(w, t) for t in range(3)]
    qs, ks, vs = [s.q for s in sts], [s.k_new for s in sts], [s.v_new for s in sts]
    # the whole problem, three steps
    rk, rv, pos = kv.ring_k.copy(), kv.ring_v.copy(), kv.pos0.copy()
    whole = [oracle.decode_step(qs[t], kv.tier1_k, kv.tier1_v, idx, rk, rv, pos, ks[t], vs[t])
             for t in range(3)]
    tasks = slice_problem(kv.tier1_k, kv.tier1_v, idx, kv.ring_k, kv.ring_v, kv.pos0,
                          qs, ks, vs, 3, workers)
    axis, _ = _slices(w.B, w.L, workers)
    parts = []
    for (t1k, t1v, sel, ring_k, ring_v, pos_s, qs_s, ks_s, vs_s, n) in tasks:
        ring_k, ring_v, pos_s = ring_k.copy(), ring_v.copy(), pos_s.copy()
        parts.append([oracle.decode_step(qs_s[t], t1k, t1v, sel, ring_k, ring_v, pos_s,
                                         ks_s[t], vs_s[t]) for t in range(n)])
    for t in range(3):
        got = np.concatenate([p[t] for p in parts], axis=0 if axis == "b" else 1)
        np.testing.assert_array_equal(got, whole[t])


def test_layer_slices_equal_the_whole_step():
    _check(WORKLOADS["tiny"].with_(L=5, B=2, W0=(128, 40)), workers=3)


def test_batch_slices_equal_the_whole_step():
    _check(WORKLOADS["tiny"].with_(B=5, L=2, W0=(0, 3, 64, 127, 128)), workers=4)
