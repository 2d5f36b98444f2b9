"""The N > 1 path of bench.py on CPU: two gloo ranks on 127.0.0.1.

The path shards by request (replicas, no data-path collective); the process
group carries only the barriers around the timed region and the max over
ranks of the elapsed time.  These tests run that logic with world_size 2 and
check the whole-job value, the disjoint request seeds, and that the reference
arm runs on rank 0 only."""

import io
import json
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _env(rank: int, world: int, port: int) -> None:
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port),
                       "WORLD_SIZE": str(world), "RANK": str(rank), "LOCAL_RANK": str(rank)})


def _timing_rank(rank: int, world: int, port: int, q) -> None:
    sys.path.insert(0, ROOT)
    _env(rank, world, port)
    import torch.distributed as dist
    import bench
    from workloads import WORKLOADS
    w_, r_, _ = bench.dist_setup(backend="gloo")
    try:
        assert (w_, r_) == (world, rank)
        bench.barrier(world)
        # each rank reports its own elapsed time; every rank must see the max
        mine = 100.0 + 50.0 * rank
        mx = bench.max_over_ranks(mine, world, torch.device("cpu"))
        w = WORKLOADS["llama3_8b"]
        seeds = bench.request_seeds(w, rank, 4)
        value = bench.job_tokens_per_s(world, 2, 4, w.B, w.T, mx)
        bench.barrier(world)
        q.put((rank, mx, seeds, value))
    finally:
        dist.destroy_process_group()


def _reference_rank(rank: int, world: int, port: int, q) -> None:
    sys.path.insert(0, ROOT)
    _env(rank, world, port)
    import bench
    buf = io.StringIO()
    with redirect_stdout(buf):
        rc = bench.main(["--impl", "reference", "--gpus", str(world), "--workload", "tiny",
                         "--steps", "1", "--warmup", "3", "--ref-step-seconds", "0.01"])
    q.put((rank, rc, buf.getvalue()))


def _run(fn, world=2):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=fn, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = [q.get(timeout=240) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    return sorted(out)


def test_two_ranks_max_time_and_job_value():
    out = _run(_timing_rank)
    (r0, mx0, seeds0, v0), (r1, mx1, seeds1, v1) = out
    assert (r0, r1) == (0, 1)
    assert mx0 == mx1 == 150.0                 # the slowest rank's time
    assert not set(seeds0) & set(seeds1)       # ranks run different requests
    # 2 ranks x 2 rounds x 4 requests x 1 sequence x 3000 steps in 150 ms
    assert v0 == v1 == pytest.approx(2 * 2 * 4 * 1 * 3000 / 0.150)


def test_reference_arm_runs_on_rank_zero_only():
    out = _run(_reference_rank)
    (r0, rc0, text0), (r1, rc1, text1) = out
    assert rc0 == 0 and rc1 == 0
    assert text1.strip() == ""
    line = json.loads(text0.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["n_gpus"] == 2
    assert line["cpu_baseline"]["kind"] == "oracle" and line["value"] > 0
    assert line["e2e"]["h2d_bytes_per_step"] == 0
