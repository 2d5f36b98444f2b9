"""Times the fp64 oracle on all host cores (bench infrastructure).

TEST / BENCH INFRASTRUCTURE ONLY, like the rest of this package: only
`bench.py`'s CPU-baseline and reference legs use it.  It does not change the
oracle: each worker process runs the unchanged `decode_step` (append, then
two-tier attention, Section 2.5) on a disjoint slice of the decode problem.
Sequences and layers are independent in a decode step (each (sequence,
layer, KV head) keeps its own ring and reads its own Tier-1 rows), so slicing
the problem along the batch or the layer axis and running the slices side by
side computes exactly the whole step.

The module imports numpy and the oracle only, so that the worker processes
(started with the "spawn" method, never forked from a process that has used
a GPU) start quickly.
"""

from __future__ import annotations

import multiprocessing as mp
import os
import time
from typing import List, Sequence, Tuple

import numpy as np

from . import cmc_oracle as _oracle


def host_cores() -> int:
    """Cores this process may run on (the affinity mask), else os.cpu_count()."""
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def _run_slice(task) -> Tuple[float, int]:
    """Runs n_steps oracle decode steps on one slice; returns (seconds, steps)."""
    (t1k, t1v, idx, ring_k, ring_v, pos, qs, ks, vs, n_steps) = task
    ring_k, ring_v, pos = ring_k.copy(), ring_v.copy(), pos.copy()
    t0 = time.perf_counter()
    for s in range(n_steps):
        p = s % len(qs)
        _oracle.decode_step(qs[p], t1k, t1v, idx, ring_k, ring_v, pos, ks[p], vs[p])
    return time.perf_counter() - t0, n_steps


def _slices(B: int, L: int, workers: int) -> Tuple[str, List[Tuple[int, int]]]:
    """Contiguous ranges of the batch axis (when B >= workers or L == 1) or of
    the layer axis, at most `workers` of them."""
    axis = "b" if (B >= workers or L == 1) else "l"
    n = B if axis == "b" else L
    parts = min(workers, n)
    bounds = [(n * i) // parts for i in range(parts + 1)]
    return axis, [(bounds[i], bounds[i + 1]) for i in range(parts)]


class HostPool:
    """A pool of `workers` spawned processes that time oracle decode steps on
    disjoint slices of one problem."""

    def __init__(self, workers: int):
        self.workers = max(1, int(workers))
        self._pool = mp.get_context("spawn").Pool(self.workers)

    def close(self):
        self._pool.close()
        self._pool.join()

    def decode_steps(self, t1k, t1v, idx, ring_k, ring_v, pos,
                     qs: Sequence[np.ndarray], ks: Sequence[np.ndarray],
                     vs: Sequence[np.ndarray], n_steps: int) -> Tuple[float, int]:
        """Runs n_steps decode steps (inputs cycled from the pools qs / ks / vs,
        each [B, L, ...]) over all slices at once.  Returns the elapsed time of
        the slowest slice (the workers run side by side) and the slice count."""
        tasks = slice_problem(t1k, t1v, idx, ring_k, ring_v, pos, qs, ks, vs, n_steps,
                              self.workers)
        results = self._pool.map(_run_slice, tasks)
        return max(r[0] for r in results), len(tasks)


def slice_problem(t1k, t1v, idx, ring_k, ring_v, pos, qs, ks, vs, n_steps: int, workers: int):
    """The worker tasks: one per contiguous range of the batch or layer axis,
    each holding that range of every tensor (and of idx / pos along the batch
    axis)."""
    B, L = ring_k.shape[0], ring_k.shape[1]
    axis, ranges = _slices(B, L, workers)
    tasks = []
    for a, b in ranges:
        if axis == "b":
            sl = (slice(a, b),)
            sel = None if idx is None else idx[a:b]
            pos_s = pos[a:b]
        else:
            sl = (slice(None), slice(a, b))
            sel = idx
            pos_s = pos
        tasks.append((t1k[sl], t1v[sl], sel, ring_k[sl], ring_v[sl], pos_s,
                      [q[sl] for q in qs], [k[sl] for k in ks], [v[sl] for v in vs],
                      n_steps))
    return tasks
