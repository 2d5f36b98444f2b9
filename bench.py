#!/usr/bin/env python3
"""Throughput benchmark of the CMC two-tier decode path on GB300.

Workload: the Llama-3-8B-shaped configuration -- batch 1, 32 layers, 32 query
/ 8 KV heads, head_dim 128, a bank of 1,024 CMEs of dimension 4,096, top-k 128,
a 512-token window, 3,000 decode steps.

One benchmark step is one generation round over R independent requests of
that shape (R = --requests, default 4): each request first runs the Tier-1
scoring + top-k selection on its own CME bank and compacts the selected K/V
rows into its dense Tier-1 cache (cmc_tier1_gather: the cache the paper's
prefill of the selected CMEs leaves), then the R requests run their 3,000
fused decode steps (ring append + two-tier attention over all 32 layers, one
launch per request per step) round-robin, request r's launches on stream
r % S (S = --streams, default 4: a server runs independent requests
concurrently; each request's steps stay in order on its stream, so a launch
of one stream overlaps the completion of another's).  `--tier1 gather` instead passes the
bank and idx to every decode step (the gather inside the attention kernel).  Each request's KV
state (84.5 MB read per step) fits in the 129 MB L2 by itself; interleaving R
requests puts (R-1) x 84.5 MB of other traffic between two steps of the same
request, so every launch reads its K/V from HBM, as it would inside a real
decoder whose weights stream through L2 between attention layers.

Reported (one JSON line on rank 0):
  value          decode tokens/s over the whole job (all ranks), selection
                 included in the timed region;
  roofline       the fused decode-step kernel: algorithmic bytes per launch
                 / average launch time, against the measured HBM copy peak;
  select_us      Tier-1 score + select per request (one launch at this
                 size), inside the benchmark step, L2-cold;
  tier1_gather_us  the once-per-request Tier-1 compaction;
  question_prologue_us, bridge_epilogue_us, denoise_us, select_stream_us
                 per call in a graph of back-to-back calls on distinct inputs
                 (at least twice the L2 per replay: every call reads HBM):
                 the question-side prologue of a request, the MemoryBridge
                 output of a bank, the denoising of a context of N * r
                 tokens, the selection alone;
  *_cold_us      one isolated call after a 512 MB write that evicts the L2
                 (median of 5; includes a launch's fixed cost);
  variant        the decode step with the other Tier-1 form, us per launch;
  e2e            the same metric through the Python API with host buffers
                 (question vector, CME bank and every step's q / new K,V
                 copied in from pinned memory, every step's output copied out,
                 by one staging-copy launch per R decode launches on each
                 stream);
  cpu_baseline   the fp64 oracle on the host, on a bounded sample.

`--impl reference` times the fp64 oracle alone on the host cores (the
reference arm; rank 0 only).
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

# The CPU oracle legs use one BLAS thread per process (the multi-core legs run
# one process per core) and say so.
for _v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, "1")

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from workloads import (WORKLOADS, context_inputs, kv_inputs, question_inputs,  # noqa: E402
                       selection_inputs, step_inputs)

METRIC = ("two-tier decode-attn tokens/s and % of 8 TB/s HBM; CME top-k select µs")
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
# machine-readable companion of profiles/decode_step_llama3_8b.md
PROFILE_FILE = os.path.join(ROOT, "profiles", "decode_step_llama3_8b.json")
# the attention launches' L2 prefetch depth for one stream of launches (the
# library's default)
SINGLE_STREAM_PREFETCH = 5
KERNEL_SOURCES = [os.path.join(ROOT, "paper_2609_25537_gb300", "csrc", f)
                  for f in ("cmc_attn.cu", "cmc_internal.cuh")]


# ----------------------------------------------------------------------------
# Accounting
# ----------------------------------------------------------------------------

def decode_step_bytes(B, L, Hq, Hkv, d, k, W, gather=False) -> int:
    """Algorithmic HBM bytes of one fused decode step with a full ring:
    k selected Tier-1 rows and W - 1 old ring rows of K and V read, the new
    token's K,V read once and written once, q read, out written, and idx
    read when the step gathers the Tier-1 rows itself."""
    kv_row = d * 2
    return (B * L * Hkv * 2 * kv_row * (k + W + 1)
            + B * L * Hq * d * 2 * 2
            + (B * k * 4 if gather else 0))


def tier1_gather_bytes(B, L, Hkv, d, k) -> int:
    """The selected K and V rows read from the bank and written densely, idx read."""
    return 2 * 2 * B * L * Hkv * k * d * 2 + B * k * 4


def decode_step_flops(B, L, Hq, d, k, W) -> int:
    """2 flops per MAC; the paper's MACs_t = 2 n_h d_h n_l L_t (appendix,
    Attention MACs Analysis) with L_t = k + W cached keys."""
    return 2 * (2 * B * Hq * d * L * (k + W))


def select_bytes(B, N, D, k) -> int:
    return 4 * B * N * D + 4 * B * D + 4 * B * k


def select_launches(B, N, D, sms) -> int:
    """Kernel launches of one cmc_score_select call with a workspace, as the
    library chooses them: one when N <= 2,048, D <= 4,096 and CTAs of R <= 8
    rows (R dividing N) cover the B N rows in one wave of one CTA per SM;
    else two (scoring, then selection)."""
    if N <= 2048 and D <= 4096:
        for R in range(8, 0, -1):
            if N % R == 0 and B * N // R <= sms:
                return 1
    return 2


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def kernel_source_hash() -> str:
    h = hashlib.sha256()
    for f in KERNEL_SOURCES:
        with open(f, "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def profiled_traffic(workload: str, tier1: str):
    """DRAM bytes per launch of the fused decode kernel from the committed ncu
    record, if it was taken on the current kernel source, for this workload
    and Tier-1 form: (in the benchmark's request loop, with L2 carried over
    between launches; one launch with L2 flushed before it), either None
    when not recorded; (None, None) otherwise."""
    try:
        with open(PROFILE_FILE) as f:
            rec = json.load(f)
        if rec["kernel_source_sha256"] != kernel_source_hash():
            return None, None
        if (rec["workload"], rec["tier1"]) != (workload, tier1):
            return None, None
        loop = rec.get("in_loop", {}).get("dram_bytes_per_launch")
        return (int(loop) if loop is not None else None), int(rec["dram_bytes_per_launch"])
    except (OSError, ValueError, KeyError, TypeError, AttributeError):
        return None, None


# ----------------------------------------------------------------------------
# Clock sampling (nvidia-smi during the timed region)
# ----------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, device: torch.device, interval_ms: int = 100):
        self.proc = None
        try:
            uuid = str(torch.cuda.get_device_properties(device).uuid)
            if not uuid.startswith("GPU-"):
                uuid = "GPU-" + uuid
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", uuid, f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", str(interval_ms)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons = [], [], set()
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for name, val in zip(self.NAMES, parts[4:8]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


# ----------------------------------------------------------------------------
# Distributed plumbing (one process per GPU; replicas only)
# ----------------------------------------------------------------------------

def dist_setup(backend: str = "nccl"):
    """One process per GPU (torchrun env vars).  The ranks run independent
    replicas of the workload (no data-path collective); the process group only
    carries the start/stop barriers and the max-over-ranks of the elapsed
    time.  `backend="gloo"` runs the same logic on CPU."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        if backend == "nccl":
            torch.cuda.set_device(local)
            dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        else:
            dist.init_process_group(backend)
    return world, rank, local


def request_seeds(w, rank: int, R: int):
    """Seeds of the R requests rank `rank` runs: distinct across ranks, so N
    ranks process N x R different requests (weak scaling)."""
    return [1000 * w.seed + 100 * rank + r for r in range(R)]


def job_tokens_per_s(world: int, K: int, R: int, B: int, T: int, max_ms: float) -> float:
    """Whole-job decode tokens/s: every rank's K rounds of R requests x B
    sequences x T steps, over the slowest rank's elapsed time."""
    return world * K * R * B * T / (max_ms / 1000.0)


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int, device) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ----------------------------------------------------------------------------
# The CPU oracle legs
# ----------------------------------------------------------------------------

def oracle_sample(w, host_state, seconds: float, min_steps: int = 1):
    """Times the oracle: one Tier-1 selection, then decode steps until
    `seconds` have passed.  Returns (decode tokens/s, steps, elapsed)."""
    import oracle
    qemb, bank, t1k, t1v, ring_k, ring_v, pos = host_state
    ring_k, ring_v, pos = ring_k.copy(), ring_v.copy(), pos.copy()
    t0 = time.perf_counter()
    idx, _ = oracle.score_select(qemb, bank, w.k)
    steps = 0
    while True:
        st = step_inputs(w, steps)
        oracle.decode_step(st.q, t1k, t1v, idx, ring_k, ring_v, pos, st.k_new, st.v_new)
        steps += 1
        el = time.perf_counter() - t0
        if steps >= min_steps and el >= seconds:
            break
    return steps * w.B / el, steps, el


def step_pool(w, n: int = 8):
    """The first n decode steps' inputs, cycled by the multi-core oracle leg
    (the GPU arm cycles a pool of the same size)."""
    sts = [step_inputs(w, t) for t in range(n)]
    return [s.q for s in sts], [s.k_new for s in sts], [s.v_new for s in sts]


def oracle_sample_parallel(w, host_state, seconds: float, step_seconds: float, pool=None):
    """Times the unchanged oracle on all host cores: one Tier-1 selection
    (one process), then decode steps run as disjoint slices of the problem
    (layers, or sequences) in a pool of spawned processes side by side, sized
    to take about `seconds` given the single-thread step time.  Returns
    (decode tokens/s, steps, elapsed, worker processes, slices)."""
    import oracle
    from oracle.host_pool import HostPool, host_cores
    qemb, bank, t1k, t1v, ring_k, ring_v, pos = host_state
    cores = host_cores()
    n_units = w.B if (w.B >= cores or w.L == 1) else w.L
    workers = max(1, min(cores, n_units))
    own = pool is None
    if own:
        pool = HostPool(workers)
    try:
        qs, ks, vs = step_pool(w)
        n_steps = max(2, int(seconds * workers / max(step_seconds, 1e-6)))
        t0 = time.perf_counter()
        idx, _ = oracle.score_select(qemb, bank, w.k)
        t_sel = time.perf_counter() - t0
        el, n_slices = pool.decode_steps(t1k, t1v, idx, ring_k, ring_v, pos, qs, ks, vs, n_steps)
    finally:
        if own:
            pool.close()
    total = t_sel + el
    return n_steps * w.B / total, n_steps, total, pool.workers, n_slices


def host_state_for(w):
    si = selection_inputs(w)
    kv = kv_inputs(w)
    return (si.question_emb, si.cme_bank, kv.tier1_k, kv.tier1_v, kv.ring_k, kv.ring_v,
            kv.pos0)


def run_reference(args, w, world, rank):
    """The reference arm: the fp64 oracle on all host cores, rank 0 only.
    Each step is one Tier-1 selection plus ~ref_step_seconds of decode steps,
    the problem's layers (or sequences) split over a pool of spawned worker
    processes; a step's time is the selection's plus the slowest worker's."""
    if rank != 0:
        return 0
    from oracle.host_pool import HostPool, host_cores
    state = host_state_for(w)
    per_step = args.ref_step_seconds
    # single-thread step time, to size each step's sample
    _, n1, el1 = oracle_sample(w, state, 0.0, min_steps=2)
    step_s = el1 / n1
    cores = host_cores()
    n_units = w.B if (w.B >= cores or w.L == 1) else w.L
    pool = HostPool(max(1, min(cores, n_units)))
    try:
        for _ in range(args.warmup):
            oracle_sample_parallel(w, state, 0.0, step_s, pool=pool)
        tokens, elapsed = 0, 0.0
        for _ in range(args.steps):
            _, steps, el, workers, n_slices = oracle_sample_parallel(w, state, per_step, step_s,
                                                                     pool=pool)
            tokens += steps * w.B
            elapsed += el
    finally:
        pool.close()
    value = tokens / elapsed
    sample = (f"per step: one Tier-1 selection + ~{per_step:g}s of fused decode steps "
              f"(all {w.L} layers) of {w.name}, split into {n_slices} slices over {workers} "
              f"worker processes; fp64 numpy, 1 BLAS thread each; host has {cores} cores")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1000.0 * elapsed / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(w, args.requests),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": workers,
                         "host_cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def workload_config(w, R):
    return {
        "workload": (f"{w.name}: B={w.B} L={w.L} Hq={w.Hq} Hkv={w.Hkv} d={w.d} "
                     f"N={w.N} D={w.D} k={w.k} W={w.W} T={w.T}"),
        "requests_round_robin": R,
        "l2": (f"inputs larger than L2: {R} independent requests interleaved, "
               f"{R * decode_step_bytes(w.B, w.L, w.Hq, w.Hkv, w.d, w.k, w.W) / 1e6:.0f} MB "
               "of KV read per round vs 129 MB L2"),
        "accumulate": "fp32",
        "parallelism": "replicas",
    }


# ----------------------------------------------------------------------------
# The GPU arm
# ----------------------------------------------------------------------------

class Request:
    """Device state of one B=1 request of the workload."""

    def __init__(self, w, dev, seed, pool, host_sel=None):
        import paper_2609_25537_gb300 as cmc
        g = torch.Generator(device=dev).manual_seed(seed)

        def randn(shape, std):
            return (torch.randn(shape, generator=g, device=dev, dtype=torch.float32)
                    * std).to(torch.bfloat16)

        B, L, Hq, Hkv, d = w.B, w.L, w.Hq, w.Hkv, w.d
        sel = host_sel if host_sel is not None else selection_inputs(w.with_(seed=seed))
        self.qemb = torch.from_numpy(sel.question_emb).to(dev)
        self.bank = torch.from_numpy(sel.cme_bank).to(dev)
        self.host_qemb = sel.question_emb
        self.host_bank = sel.cme_bank
        self.t1k = randn((B, L, Hkv, w.N, d), w.kv_std)
        self.t1v = randn((B, L, Hkv, w.N, d), w.kv_std)
        self.ring_k = randn((B, L, Hkv, w.W, d), w.kv_std)
        self.ring_v = randn((B, L, Hkv, w.W, d), w.kv_std)
        self.pos = torch.full((B,), w.W, dtype=torch.int64, device=dev)
        self.q = randn((pool, B, L, Hq, d), w.q_std)
        self.k_new = randn((pool, B, L, Hkv, d), w.kv_std)
        self.v_new = randn((pool, B, L, Hkv, d), w.kv_std)
        self.idx = torch.empty((B, w.k), dtype=torch.int32, device=dev)
        self.t1k_dense = torch.empty((B, L, Hkv, w.k, d), dtype=torch.bfloat16, device=dev)
        self.t1v_dense = torch.empty((B, L, Hkv, w.k, d), dtype=torch.bfloat16, device=dev)
        self.out = torch.empty((B, L, Hq, d), dtype=torch.bfloat16, device=dev)
        # zero-filled once: the selection's completion counters start at zero
        self.sel_ws = torch.zeros(cmc.score_select_workspace_size(B, w.N), dtype=torch.uint8,
                                  device=dev)
        self.ws = cmc.DecodeWorkspace(cmc.dims_of(self.out, self.t1k, self.idx, self.ring_k),
                                      dev)
        self.ws_dense = cmc.DecodeWorkspace(
            cmc.dims_of(self.out, self.t1k_dense, None, self.ring_k), dev)

    def select(self):
        import paper_2609_25537_gb300 as cmc
        cmc.score_select(self.qemb, self.bank, self.idx.shape[1], idx_out=self.idx,
                         workspace=self.sel_ws)

    def gather(self):
        import paper_2609_25537_gb300 as cmc
        cmc.tier1_gather(self.t1k, self.t1v, self.idx, out_k=self.t1k_dense,
                         out_v=self.t1v_dense, workspace=self.ws_dense)

    def decode(self, p, q=None, k_new=None, v_new=None, mode="dense", rope=False, out=None):
        """One fused decode step; with `rope` the GQA-layer step that rotates
        q and k_new (theta 5e5, the Llama-3 base; positions after the k
        Tier-1 rows)."""
        import paper_2609_25537_gb300 as cmc
        q = self.q[p] if q is None else q
        k_new = self.k_new[p] if k_new is None else k_new
        v_new = self.v_new[p] if v_new is None else v_new
        out = self.out if out is None else out
        kw = dict(rope_theta=500000.0, rope_offset=self.idx.shape[1]) if rope else {}
        if mode == "dense":
            cmc.decode_step(q, self.t1k_dense, self.t1v_dense, None, self.ring_k, self.ring_v,
                            self.pos, k_new, v_new, out=out, workspace=self.ws_dense, **kw)
        else:
            cmc.decode_step(q, self.t1k, self.t1v, self.idx, self.ring_k, self.ring_v,
                            self.pos, k_new, v_new, out=out, workspace=self.ws, **kw)

    def host_state(self):
        def bits(t):
            return t.view(torch.int16).cpu().numpy().view(np.uint16)
        return (self.host_qemb, self.host_bank, bits(self.t1k), bits(self.t1v),
                bits(self.ring_k), bits(self.ring_v), self.pos.cpu().numpy().copy())


def run_gpu(args, w, world, rank, local):
    import paper_2609_25537_gb300 as cmc
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    cmc.lib()  # fails loudly when the library is not built

    R, T, P = args.requests, args.decode_steps, args.pool
    if T % P:
        raise SystemExit(f"--decode-steps {T} must be a multiple of --pool {P}")
    sel0 = selection_inputs(w)
    reqs = [Request(w, dev, seed, P, host_sel=sel0 if (r == 0 and rank == 0) else None)
            for r, seed in enumerate(request_seeds(w, rank, R))]
    torch.cuda.synchronize(dev)  # state was created on the default stream
    want_cpu = rank == 0 and world == 1 and not args.no_cpu_baseline
    # the oracle's copy of request 0, taken before any kernel of ours touches it
    cpu_state = reqs[0].host_state() if want_cpu else None
    stream = torch.cuda.Stream(device=dev)
    # the decode launches of the R independent requests go to S streams
    # (request r to stream r % S), as a server runs independent requests
    # concurrently; every request's steps stay in order on its stream
    S = max(1, min(args.streams, R))
    streams = [stream] + [torch.cuda.Stream(device=dev) for _ in range(S - 1)]
    # the attention launches' L2 prefetch depth before their grid dependency
    # wait: the library's default suits one stream of launches; with the
    # requests on several streams (launches already overlapping) none
    # measured best at the Llama shape (11.92 us per launch against 12.89)
    pf = args.l2_prefetch if args.l2_prefetch >= 0 else (0 if S > 1 else SINGLE_STREAM_PREFETCH)
    cmc.set_l2_prefetch_tiles(pf)

    mode = args.tier1
    other = "gather" if mode == "dense" else "dense"
    # eager warm-up of every kernel before graph capture
    with torch.cuda.stream(stream):
        for r in reqs:
            r.select()
            r.gather()
            r.decode(0, mode=mode)
            r.decode(0, mode=other)
            r.decode(0, mode=mode, rope=True)
    stream.synchronize()

    # one graph = GR rounds of R decode launches (forked over the S streams
    # and joined again at its end; round p takes the pool's input p % P),
    # replayed T / GR times per step; GR = P by default (8 rounds measured
    # faster than 24 or 40 at the Llama shape)
    GR = args.graph_rounds or P
    if T % GR or GR % P:
        raise SystemExit(f"--graph-rounds {GR} must divide --decode-steps {T} and be a "
                         f"multiple of --pool {P}")

    def capture(m, rope=False):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for st in streams[1:]:
                st.wait_stream(stream)
            for p in range(GR):
                for ri, r in enumerate(reqs):
                    with torch.cuda.stream(streams[ri % S]):
                        r.decode(p % P, mode=m, rope=rope)
            for st in streams[1:]:
                stream.wait_stream(st)
        return g
    graph = capture(mode)
    replays = T // GR

    # the once-per-request kernels, also as graphs (so that their times are
    # GPU times, not Python launch rates)
    def capture_calls(fn):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for r in reqs:
                fn(r)
        return g
    g_sel = capture_calls(lambda r: r.select())
    g_gat = capture_calls(lambda r: r.gather()) if mode == "dense" else None

    def one_step(ev=None):
        with torch.cuda.stream(stream):
            if ev is not None:
                ev[0].record(stream)
            g_sel.replay()
            if ev is not None:
                ev[1].record(stream)
            if g_gat is not None:
                g_gat.replay()
            if ev is not None:
                ev[2].record(stream)
            for _ in range(replays):
                graph.replay()
            if ev is not None:
                ev[3].record(stream)

    for _ in range(args.warmup):
        one_step()
    stream.synchronize()

    K = args.steps
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(K)]
    barrier(world)
    torch.cuda.synchronize(dev)
    clocks = ClockSampler(dev) if rank == 0 else None
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for s in range(K):
        one_step(evs[s])
    t_end.record(stream)
    torch.cuda.synchronize(dev)
    barrier(world)
    clk = clocks.stop() if clocks is not None else None

    elapsed_ms = t_start.elapsed_time(t_end)
    sel_ms = [e[0].elapsed_time(e[1]) for e in evs]
    gat_ms = [e[1].elapsed_time(e[2]) for e in evs]
    dec_ms = [e[2].elapsed_time(e[3]) for e in evs]
    max_ms = max_over_ranks(elapsed_ms, world, dev)
    value = job_tokens_per_s(world, K, R, w.B, T, max_ms)

    launches_dec = K * R * T
    # kernels per fused decode call (attention, plus combine after a stream-K split)
    step_ctas, step_launches = cmc.decode_attn_plan(
        cmc.dims_of(reqs[0].out, reqs[0].t1k_dense if mode == "dense" else reqs[0].t1k,
                    None if mode == "dense" else reqs[0].idx, reqs[0].ring_k), fused=True)
    n_units = w.B * w.L * w.Hkv
    if step_launches > 1:
        plan_txt = " + two_tier_combine_kernel (units split between CTAs)"
    elif step_ctas > n_units:
        plan_txt = (f" (clusters of {step_ctas // n_units} CTAs per unit, merged in distributed "
                    "shared memory; one launch)")
    elif step_ctas < n_units:
        plan_txt = " (whole units per CTA; one launch)"
    else:
        plan_txt = " (one CTA per unit; one launch)"
    launch_us = 1000.0 * sum(dec_ms) / launches_dec
    nbytes = decode_step_bytes(w.B, w.L, w.Hq, w.Hkv, w.d, w.k, w.W, gather=mode == "gather")
    achieved = nbytes / (launch_us * 1e-6) / 1e9
    peak, peak_kind = measured_peaks()
    select_us = 1000.0 * statistics.median(sel_ms) / R
    gather_us = 1000.0 * statistics.median(gat_ms) / R if mode == "dense" else 0.0

    def time_graph(g, launches):
        with torch.cuda.stream(stream):
            g.replay()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(args.variant_replays):
                g.replay()
            e1.record(stream)
        stream.synchronize()
        return 1000.0 * e0.elapsed_time(e1) / (args.variant_replays * launches)

    # the decode step with the other Tier-1 form, and the GQA-layer step with
    # rotary embedding (same state, same launch shape)
    variant = rope_variant = warm_l2 = None
    if not args.no_variant:
        g2 = capture(other)
        v_us = time_graph(g2, GR * R)
        v_bytes = decode_step_bytes(w.B, w.L, w.Hq, w.Hkv, w.d, w.k, w.W,
                                    gather=other == "gather")
        variant = {"tier1": other, "us_per_launch": v_us,
                   "achieved_gbs": v_bytes / (v_us * 1e-6) / 1e9}
        del g2
        g3 = capture(mode, rope=True)
        r_us = time_graph(g3, GR * R)
        rope_variant = {"step": "GQA layer: rotary embedding of q and k_new + append + attention",
                        "tier1": mode, "us_per_launch": r_us,
                        "achieved_gbs": nbytes / (r_us * 1e-6) / 1e9}
        del g3
        # warm-L2 companion: one request's launches back to back, so its K/V
        # (84.5 MB at the Llama shape) stays in the 129 MB L2 between launches
        cmc.set_l2_prefetch_tiles(SINGLE_STREAM_PREFETCH)  # one stream of launches
        gw = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gw, stream=stream):
            for p in range(P * R):
                reqs[0].decode(p % P, mode=mode)
        cmc.set_l2_prefetch_tiles(pf)
        w_us = time_graph(gw, P * R)
        warm_l2 = {"requests": 1, "us_per_launch": w_us,
                   "achieved_gbs": nbytes / (w_us * 1e-6) / 1e9,
                   "note": "one request's K/V re-read every launch (L2-resident when it "
                           "fits); not the headline, which reads HBM"}
        del gw

    # Once-per-request kernels outside the decode loop.  Each is timed as a
    # graph of back-to-back calls on distinct copies of its inputs -- enough
    # copies that the calls of one replay read at least twice the L2 (129 MB),
    # so every call reads HBM -- replayed after warm-up; per call = replay
    # time / calls (a call's launch is amortised and, under programmatic
    # dependent launch, overlaps the one before: the device-side cost of a
    # stream of requests).  The bank-sized ones also report one isolated call
    # after a 512 MB write that evicts the L2 (median of 5), which includes a
    # launch's fixed cost of several microseconds.
    flush = torch.empty(512 << 20, dtype=torch.uint8, device=dev)

    def cold_us(fn, reps=5):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(stream):
            fn()  # warm-up outside capture
        stream.synchronize()
        with torch.cuda.graph(g, stream=stream):
            fn()
        times = []
        with torch.cuda.stream(stream):
            for _ in range(reps + 1):
                flush.zero_()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                g.replay()
                e1.record(stream)
                times.append((e0, e1))
        stream.synchronize()
        return 1000.0 * statistics.median(a.elapsed_time(b) for a, b in times[1:])

    def stream_us(fns, reps=10):
        with torch.cuda.stream(stream):
            for fn in fns:
                fn()  # warm-up outside capture
        stream.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for fn in fns:
                fn()
        with torch.cuda.stream(stream):
            for _ in range(3):
                g.replay()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(reps):
                g.replay()
            e1.record(stream)
        stream.synchronize()
        return 1000.0 * e0.elapsed_time(e1) / (reps * len(fns))

    def copies_for(nbytes):
        return max(2, min(16, -(-2 * 129_000_000 // max(nbytes, 1))))

    prologue_us = bridge_us = denoise_us = select_cold_us = batched = None
    prologue_cold_us = bridge_cold_us = None
    denoise_bytes = 0
    if not args.no_variant:
        # the question-side prologue of one request (pool q_vec, score + select,
        # CME-guided window start)
        qi = question_inputs(w, sel0, ratio=8 if w.N >= 16384 else 4)
        tok = torch.from_numpy(qi.tokens).to(dev)
        qlen = torch.from_numpy(qi.q_len).to(dev)
        offs = torch.from_numpy(qi.chunk_offset).to(dev)
        clen = torch.from_numpy(qi.ctx_len).to(dev)
        r0 = reqs[0]
        nc = copies_for(r0.bank.numel() * 4)
        banks = [r0.bank] + [r0.bank.clone() for _ in range(nc - 1)]
        toks = [tok] + [tok.clone() for _ in range(nc - 1)]
        ws_qs = [torch.zeros(cmc.lib().cmc_question_select_workspace_size(w.B, w.N),
                             dtype=torch.uint8, device=dev) for _ in range(nc)]
        ws_ss = [torch.zeros(cmc.score_select_workspace_size(w.B, w.N), dtype=torch.uint8,
                             device=dev) for _ in range(nc)]
        idxs = [torch.empty_like(r0.idx) for _ in range(nc)]
        # the selection alone, timed the same ways
        select_cold_us = cold_us(lambda: cmc.score_select(r0.qemb, r0.bank, w.k, idx_out=r0.idx,
                                                          workspace=r0.sel_ws))
        sel_stream_us = stream_us([
            (lambda i=i: cmc.score_select(r0.qemb, banks[i], w.k, idx_out=idxs[i],
                                          workspace=ws_ss[i])) for i in range(nc)])
        prologue_cold_us = cold_us(lambda: cmc.question_select(
            tok, r0.bank, w.k, q_len=qlen, chunk_offset=offs, ctx_len=clen, W=w.W,
            workspace=ws_qs[0]))
        prologue_us = stream_us([
            (lambda i=i: cmc.question_select(toks[i], banks[i], w.k, q_len=qlen,
                                             chunk_offset=offs, ctx_len=clen, W=w.W,
                                             workspace=ws_qs[i])) for i in range(nc)])
        # MemoryBridge output (LayerNorm, nu tanh, norm cap) on a bank-sized
        # MLP output, out of place
        outs = [torch.empty_like(r0.bank) for _ in range(nc)]
        bridge_cold_us = cold_us(lambda: cmc.bridge_epilogue(banks[0], 0.8, out=outs[0]))
        bridge_us = stream_us([(lambda i=i: cmc.bridge_epilogue(banks[i], 0.8, out=outs[i]))
                               for i in range(nc)])
        del outs, banks, toks
        # graph-based denoising of one context of |C| = N * r tokens (H = 1280,
        # GPT2-Large's width; g = 3, tau = 0.05, keep-minimum 16)
        ratio = 8 if w.N >= 16384 else 4
        if args.denoise_tokens:
            ratio = max(1, args.denoise_tokens // w.N)
        ci = context_inputs(w.with_(B=1), H=1280, ratio=ratio)
        emb = torch.from_numpy(ci.emb).to(dev)
        denoise_bytes = emb.numel() * 4
        nd = copies_for(denoise_bytes)
        embs = [emb] + [emb.clone() for _ in range(nd - 1)]
        ws_ds = [torch.zeros(cmc.lib().cmc_denoise_workspace_size(1, emb.shape[1]),
                             dtype=torch.uint8, device=dev) for _ in range(nd)]
        denoise_us = stream_us([(lambda i=i: cmc.denoise(embs[i], workspace=ws_ds[i]))
                                for i in range(nd)])
        del emb, embs
        if w.B == 1:
            # the same calls with the inputs of RB requests in each (B = RB), as
            # a server that batches arriving requests would issue them; per
            # request = per call / RB, back to back on distinct inputs
            RB = 4
            wb = w.with_(B=RB)
            sib = selection_inputs(wb)
            qb = torch.from_numpy(sib.question_emb).to(dev)
            bb = torch.from_numpy(sib.cme_bank).to(dev)
            nb = copies_for(bb.numel() * 4)
            bbs = [bb] + [bb.clone() for _ in range(nb - 1)]
            wsb = [torch.zeros(cmc.score_select_workspace_size(RB, w.N), dtype=torch.uint8,
                               device=dev) for _ in range(nb)]
            sel_b = stream_us([(lambda i=i: cmc.score_select(qb, bbs[i], w.k, workspace=wsb[i]))
                               for i in range(nb)]) / RB
            qib = question_inputs(wb, sib, ratio=ratio)
            tkb = torch.from_numpy(qib.tokens).to(dev)
            tkbs = [tkb] + [tkb.clone() for _ in range(nb - 1)]
            qlb = torch.from_numpy(qib.q_len).to(dev)
            ofb = torch.from_numpy(qib.chunk_offset).to(dev)
            clb = torch.from_numpy(qib.ctx_len).to(dev)
            wqb = [torch.zeros(cmc.lib().cmc_question_select_workspace_size(RB, w.N),
                               dtype=torch.uint8, device=dev) for _ in range(nb)]
            pro_b = stream_us([(lambda i=i: cmc.question_select(
                tkbs[i], bbs[i], w.k, q_len=qlb, chunk_offset=ofb, ctx_len=clb, W=w.W,
                workspace=wqb[i])) for i in range(nb)]) / RB
            outs = [torch.empty_like(bb) for _ in range(nb)]
            br_b = stream_us([(lambda i=i: cmc.bridge_epilogue(bbs[i], 0.8, out=outs[i]))
                              for i in range(nb)]) / RB
            del outs, bbs, tkbs
            cib = context_inputs(wb, H=1280, ratio=ratio)
            eb = torch.from_numpy(cib.emb).to(dev)
            ntb = torch.from_numpy(cib.n_tokens).to(dev)
            tok_bytes = int(cib.n_tokens.sum()) * cib.emb.shape[2] * 4
            ndb = copies_for(eb.numel() * 4)
            ebs = [eb] + [eb.clone() for _ in range(ndb - 1)]
            wsd = [torch.zeros(cmc.lib().cmc_denoise_workspace_size(RB, eb.shape[1]),
                               dtype=torch.uint8, device=dev) for _ in range(ndb)]
            dn_b = stream_us([(lambda i=i: cmc.denoise(ebs[i], n_tokens=ntb, workspace=wsd[i]))
                              for i in range(ndb)]) / RB
            del ebs
            bank_bytes = 4 * w.N * w.D
            batched = {
                "requests_per_call": RB,
                "note": "per request, calls of RB requests back to back on distinct inputs",
                "select_us": sel_b, "select_gbs": bank_bytes / (sel_b * 1e-6) / 1e9,
                "question_prologue_us": pro_b,
                "bridge_epilogue_us": br_b, "bridge_epilogue_gbs": 2 * bank_bytes / (br_b * 1e-6) / 1e9,
                "denoise_us": dn_b, "denoise_gbs": tok_bytes / RB / (dn_b * 1e-6) / 1e9,
                "denoise_tokens": [int(x) for x in cib.n_tokens]}
    del flush

    # e2e through the Python API with pinned host buffers
    e2e = run_e2e(args, w, reqs, dev, stream, world, streams) if not args.no_e2e else None

    # CPU oracle baseline (rank 0, N = 1)
    cpu = None
    if want_cpu:
        from oracle.host_pool import host_cores
        tps1, steps1, el1 = oracle_sample(w, cpu_state, args.cpu_seconds)
        tps, steps, el, workers, n_slices = oracle_sample_parallel(
            w, cpu_state, args.cpu_seconds, el1 / steps1)
        cpu = {"value": tps, "unit": "tokens/s", "cores": workers, "host_cores": host_cores(),
               "kind": "oracle",
               "sample": (f"one Tier-1 selection + {steps} fused decode steps (all {w.L} "
                          f"layers) of {w.name} in {el:.1f}s, the step split into {n_slices} "
                          f"slices run side by side in {workers} spawned worker processes "
                          "(fp64 numpy, 1 BLAS thread each)"),
               "single_thread": {"value": tps1, "unit": "tokens/s", "cores": 1,
                                 "sample": (f"one Tier-1 selection + {steps1} fused decode "
                                            f"steps in {el1:.1f}s, one process")}}

    if rank != 0:
        return 0
    # DRAM bytes per launch from the committed ncu record: in the request loop
    # (L2 carried over between launches: part of a request's K/V survives the
    # other requests' traffic) and with L2 flushed
    traffic_loop, traffic_cold = profiled_traffic(w.name, mode)
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
        "steps": K, "warmup": args.warmup, "ms_per_step": max_ms / K,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic",
        "config": dict(workload_config(w, R), tier1=mode),
        "tier1": mode,
        "decode_streams": S,
        "l2_prefetch_tiles": pf,
        "decode_us_per_launch": launch_us,
        "hbm_pct_of_8tbs": 100.0 * achieved / NOMINAL_HBM_GBS,
        "select_us": select_us,
        "select_cold_us": select_cold_us,
        "select_stream_us": sel_stream_us if not args.no_variant else None,
        "question_prologue_us": prologue_us,
        "question_prologue_cold_us": prologue_cold_us,
        "bridge_epilogue_cold_us": bridge_cold_us,
        "bridge_epilogue_us": bridge_us,
        "bridge_epilogue_gbs": (8 * w.B * w.N * w.D / (bridge_us * 1e-6) / 1e9
                                if bridge_us else None),
        "denoise_us": denoise_us,
        "denoise_gbs": denoise_bytes / (denoise_us * 1e-6) / 1e9 if denoise_us else None,
        "tier1_gather_us": gather_us,
        "tier1_gather_gbs": (tier1_gather_bytes(w.B, w.L, w.Hkv, w.d, w.k) / (gather_us * 1e-6)
                             / 1e9 if gather_us > 0 else None),
        "batched_requests": batched,
        "variant": variant,
        "rope_variant": rope_variant,
        "warm_l2": warm_l2,
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "peak_kind": f"hbm copy, {peak_kind}",
                     "kernel": (f"fused decode step: two_tier_attn_kernel<{w.d},{w.Hq // w.Hkv},fused,3>"
                                + plan_txt),
                     "bytes_per_launch": nbytes, "traffic": traffic_loop,
                     "traffic_cold": traffic_cold,
                     "flops_per_launch": decode_step_flops(w.B, w.L, w.Hq, w.d, w.k, w.W)},
        "select_roofline": {"bound": "hbm", "bytes": select_bytes(w.B, w.N, w.D, w.k),
                            "achieved": select_bytes(w.B, w.N, w.D, w.k) / (select_us * 1e-6)
                            / 1e9, "unit": "GB/s"},
        "e2e": e2e,
        "cpu_baseline": cpu,
        # per request and step: the selection, the compaction (dense Tier-1)
        # and T fused decode calls
        "gpu_launches": K * R * (T * step_launches + (1 if mode == "dense" else 0)
                                 + select_launches(w.B, w.N, w.D, torch.cuda.get_device_properties(
                                     dev).multi_processor_count)),
        "clocks": clk,
    }
    print(json.dumps(line), flush=True)
    return 0


def run_e2e(args, w, reqs, dev, stream, world, streams):
    """Same metric through the public Python API with host buffers: the
    question vector and CME bank of each request and, every decode step, q and
    the new token's K,V are copied in from pinned host memory and the output
    copied back to pinned host memory.  The requests are split over the same
    streams as the device-resident loop (request r on stream r % S), each
    stream a serving loop of its own: every scheduling round (one decode step
    of each of its requests) moves their inputs in together, and a round's
    outputs go out together -- one staging-copy launch per round
    (cmc.stage_copies) on that stream carries the inputs of this round and the
    outputs of the round two back.  It copies without waiting for the decode
    before it (inputs double-buffered, outputs triple-buffered, so that decode
    never touches what it copies) and completes after it, so every decode
    launch keeps programmatic dependent launch and the copies overlap decode
    work.  60 rounds (12, 6 or 2 when T is not a multiple of 60) are captured
    in one CUDA graph; the buffers rotate across replays, so a replay's first two
    copy launches carry the previous replay's last two rounds' outputs, and
    one copy launch after the step's last replay the step's last two.
    Selection and compaction run eagerly."""
    import paper_2609_25537_gb300 as cmc
    R, T, P0 = args.requests, args.decode_steps, args.pool
    S = len(streams)
    groups = [[i for i in range(R) if i % S == j] for j in range(S)]
    # a stream's staging copy carries `spr` rounds of its requests (one by
    # default: with one request a stream, one copy launch per decode launch
    # measured faster than one per two or four)
    spr = max(1, args.e2e_copy_rounds)
    # rounds per graph: a multiple of 6 super-rounds of spr rounds when T
    # allows, so that the double-buffered inputs and triple-buffered outputs
    # continue across replays and only the step's last two need a copy after
    # the last replay; 60 rounds when T allows (74.1-74.2 k tokens/s at the
    # Llama shape against 72.7 k with 12; 120 or 300: 74.4 k)
    P = next((c for c in (60 * spr, 12 * spr, 6 * spr, 2 * spr) if T % c == 0), None)
    if P is None:  # one round per copy
        spr = 1
        P = next(c for c in (12, 6, P0, 2, T) if T % c == 0)
    Q = P // spr  # super-rounds per graph (>= 2 unless T = 1)
    rotate = Q % 6 == 0
    steps = max(1, min(args.steps, args.e2e_steps))
    nq, nk = reqs[0].q[0].numel(), reqs[0].k_new[0].numel()
    per_req = nq + 2 * nk
    out_shape = tuple(reqs[0].out.shape)
    # per stream: host round p holds its requests' packed (q, k_new, v_new) of
    # step p (the pool's P0 inputs, cycled); device buffers of one super-round
    host_in, host_out, in_d, out_d = [], [], [], []
    for grp in groups:
        host_in.append(torch.cat([torch.cat([reqs[i].q.reshape(P0, -1), reqs[i].k_new.reshape(P0, -1),
                                             reqs[i].v_new.reshape(P0, -1)], dim=1) for i in grp],
                                 dim=1)[[p % P0 for p in range(P)]].cpu().contiguous().pin_memory())
        host_out.append(torch.empty((P, len(grp)) + out_shape, dtype=torch.bfloat16).pin_memory())
        in_d.append([torch.empty(spr * len(grp) * per_req, dtype=torch.bfloat16, device=dev)
                     for _ in range(2)])
        out_d.append([torch.empty((spr, len(grp)) + out_shape, dtype=torch.bfloat16, device=dev)
                      for _ in range(3)])
    host_sel = [(r.qemb.cpu().pin_memory(), r.bank.cpu().pin_memory()) for r in reqs]

    def views(gi, par, j, k):
        i = groups[gi][k]
        base = in_d[gi][par][(j * len(groups[gi]) + k) * per_req:(j * len(groups[gi]) + k + 1) * per_req]
        return (base[:nq].view(reqs[i].q[0].shape), base[nq:nq + nk].view(reqs[i].k_new[0].shape),
                base[nq + nk:].view(reqs[i].v_new[0].shape))

    def fork():
        for st in streams[1:]:
            st.wait_stream(stream)

    def join():
        for st in streams[1:]:
            stream.wait_stream(st)

    def rows(sr):  # host rows of super-round sr
        return slice(sr * spr, (sr + 1) * spr)

    def last_two():  # the outputs of the last two super-rounds, after every decode
        fork()
        for gi in range(S):
            with torch.cuda.stream(streams[gi]):
                cmc.stage_copies([(out_d[gi][(Q - 2) % 3], host_out[gi][rows(Q - 2)]),
                                  (out_d[gi][(Q - 1) % 3], host_out[gi][rows(Q - 1)])],
                                 wait_first=True, device=dev)
        join()

    def rounds():
        fork()
        for sr in range(Q):
            for gi, grp in enumerate(groups):
                with torch.cuda.stream(streams[gi]):
                    pairs = [(host_in[gi][rows(sr)], in_d[gi][sr % 2])]
                    if sr >= 2 or rotate:  # super-rounds 0, 1: the previous replay's last two
                        pairs.append((out_d[gi][(sr - 2) % 3], host_out[gi][rows((sr - 2) % Q)]))
                    cmc.stage_copies(pairs, device=dev)
                    for j in range(spr):
                        for k, i in enumerate(grp):
                            q, kn, vn = views(gi, sr % 2, j, k)
                            reqs[i].decode((sr * spr + j) % P0, q=q, k_new=kn, v_new=vn,
                                           mode=args.tier1, out=out_d[gi][sr % 3][j, k])
        join()
        if not rotate:
            last_two()

    graph = None
    try:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            rounds()
        graph = g
    except Exception as e:  # capture unsupported here: run the same calls eagerly
        print(f"e2e: graph capture failed ({type(e).__name__}: {e}); eager loop", file=sys.stderr)
        torch.cuda.synchronize(dev)

    def step():
        with torch.cuda.stream(stream):
            for r, (hq, hb) in zip(reqs, host_sel):
                r.qemb.copy_(hq, non_blocking=True)
                r.bank.copy_(hb, non_blocking=True)
                cmc.score_select(r.qemb, r.bank, w.k, idx_out=r.idx, workspace=r.sel_ws)
                if args.tier1 == "dense":
                    r.gather()
            for _ in range(T // P):
                if graph is not None:
                    graph.replay()
                else:
                    rounds()
            if rotate:
                last_two()
        stream.synchronize()

    step()  # warm-up
    barrier(world)
    t0 = time.perf_counter()
    for _ in range(steps):
        step()
    el = time.perf_counter() - t0
    el = max_over_ranks(el, world, dev)
    h2d = R * (reqs[0].qemb.numel() * 4 + reqs[0].bank.numel() * 4) + T * R * per_req * 2
    d2h = R * T * reqs[0].out.numel() * 2
    return {"value": world * steps * R * w.B * T / el, "unit": "tokens/s",
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": steps,
            "per_step_graph": graph is not None, "streams": S,
            "copies": ("per round of decode steps of each stream's requests, one staging-copy "
                       "launch on that stream: this round's inputs in, the outputs of the "
                       "round two back out")}


def run_ablation(args, dev):
    """The ablation sweep on the Llama-3-8B head shape (one layer, bank of
    1,024 CMEs): for every (k, W, B) of the grid, the fused decode step over a
    dense Tier-1 cache of k rows (idx passed instead when k = 0: Tier-1 empty)
    and a full ring of W slots, timed as CUDA graphs of 8 rounds of R requests
    round-robin, R chosen so that R steps read at least 2 x 129 MB (at most
    8; smaller points are L2-resident and latency-bound, and say so).  Inputs
    are seeded Gaussian bf16 drawn on the device.  One JSON line."""
    import paper_2609_25537_gb300 as cmc
    from workloads.configs import ABLATION_B, ABLATION_K, ABLATION_W, ablation_workload
    torch.cuda.set_device(dev)
    cmc.lib()
    stream = torch.cuda.Stream(device=dev)
    peak, peak_kind = measured_peaks()
    P, reps = 8, 20
    rows = []
    for k in ABLATION_K:
        for W in ABLATION_W:
            for B in ABLATION_B:
                w = ablation_workload(k, W, B)
                nbytes = decode_step_bytes(w.B, w.L, w.Hq, w.Hkv, w.d, w.k, w.W,
                                           gather=w.k == 0)
                R = max(1, min(8, -(-2 * 129_000_000 // nbytes)))
                g = torch.Generator(device=dev).manual_seed(4)

                def randn(shape, std):
                    return (torch.randn(shape, generator=g, device=dev) * std).to(torch.bfloat16)
                reqs = []
                for _ in range(R):
                    kk = max(w.k, 1)
                    st = {
                        "t1k": randn((B, 1, w.Hkv, kk, w.d), w.kv_std),
                        "t1v": randn((B, 1, w.Hkv, kk, w.d), w.kv_std),
                        "idx": (torch.empty((B, 0), dtype=torch.int32, device=dev) if w.k == 0
                                else None),
                        "ring_k": randn((B, 1, w.Hkv, W, w.d), w.kv_std),
                        "ring_v": randn((B, 1, w.Hkv, W, w.d), w.kv_std),
                        "pos": torch.full((B,), W, dtype=torch.int64, device=dev),
                        "q": randn((P, B, 1, w.Hq, w.d), w.q_std),
                        "kn": randn((P, B, 1, w.Hkv, w.d), w.kv_std),
                        "vn": randn((P, B, 1, w.Hkv, w.d), w.kv_std),
                        "out": torch.empty((B, 1, w.Hq, w.d), dtype=torch.bfloat16, device=dev),
                    }
                    st["ws"] = cmc.DecodeWorkspace(
                        cmc.dims_of(st["out"], st["t1k"], st["idx"], st["ring_k"]), dev)
                    reqs.append(st)

                def call(st, p):
                    cmc.decode_step(st["q"][p], st["t1k"], st["t1v"], st["idx"], st["ring_k"],
                                    st["ring_v"], st["pos"], st["kn"][p], st["vn"][p],
                                    out=st["out"], workspace=st["ws"])
                with torch.cuda.stream(stream):
                    for st in reqs:
                        call(st, 0)
                stream.synchronize()
                gr = torch.cuda.CUDAGraph()
                with torch.cuda.graph(gr, stream=stream):
                    for p in range(P):
                        for st in reqs:
                            call(st, p)
                with torch.cuda.stream(stream):
                    for _ in range(3):
                        gr.replay()
                    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    e0.record(stream)
                    for _ in range(reps):
                        gr.replay()
                    e1.record(stream)
                stream.synchronize()
                us = 1000.0 * e0.elapsed_time(e1) / (reps * P * R)
                ctas, launches = cmc.decode_attn_plan(
                    cmc.dims_of(reqs[0]["out"], reqs[0]["t1k"], reqs[0]["idx"], reqs[0]["ring_k"]))
                gbs = nbytes / (us * 1e-6) / 1e9
                rows.append({"k": k, "W": W, "B": B, "bytes_per_step": nbytes, "requests": R,
                             "l2": "resident" if R * nbytes < 129_000_000 else "larger than L2",
                             "us_per_step": round(us, 3), "achieved_gbs": round(gbs, 1),
                             "frac": round(gbs / peak, 4), "ctas": ctas, "launches": launches})
                del reqs, gr
    print(json.dumps({"ablation": rows, "peak_gbs": peak, "peak_kind": peak_kind,
                      "shape": "Llama-3-8B heads (32 q / 8 KV, d = 128), one layer, bank of 1,024 CMEs",
                      "tier1": "dense (k = 0: none)"}), flush=True)
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=("cmc", "reference"), default="cmc")
    ap.add_argument("--workload", default="llama3_8b", choices=sorted(WORKLOADS))
    ap.add_argument("--requests", type=int, default=4)
    ap.add_argument("--decode-steps", type=int, default=None)
    ap.add_argument("--pool", type=int, default=8)
    ap.add_argument("--graph-rounds", type=int, default=0,
                    help="decode rounds per CUDA graph of the device loop (0: --pool); a "
                         "multiple of --pool dividing the decode steps")
    ap.add_argument("--l2-prefetch", type=int, default=-1,
                    help="K/V tiles per CTA the attention launches prefetch into L2 before "
                         "their grid dependency wait (-1: 0 with several streams, else 5)")
    ap.add_argument("--streams", type=int, default=4,
                    help="streams the independent requests' decode launches are spread over")
    ap.add_argument("--e2e-steps", type=int, default=2)
    ap.add_argument("--e2e-copy-rounds", type=int, default=1,
                    help="rounds (one decode step of each of a stream's requests) that each "
                         "staging copy of the e2e loop carries")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--tier1", choices=("dense", "gather"), default="dense",
                    help="Tier-1 form of the timed decode steps")
    ap.add_argument("--no-variant", action="store_true")
    ap.add_argument("--variant-replays", type=int, default=20)
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--ref-step-seconds", type=float, default=2.0)
    ap.add_argument("--ablation", action="store_true",
                    help="time the fused decode step over the k x W x B ablation grid instead")
    ap.add_argument("--denoise-tokens", type=int, default=0,
                    help="tokens of the denoised context (default N x 4, N x 8 for N >= 16384)")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        raise SystemExit("--warmup must be >= 3")
    w = WORKLOADS[args.workload]
    if args.decode_steps is None:
        args.decode_steps = w.T
    world, rank, local = dist_setup() if args.impl == "cmc" else (
        int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")), 0)
    if world != args.gpus and rank == 0:
        print(f"warning: --gpus {args.gpus} but WORLD_SIZE {world}", file=sys.stderr)
    if args.ablation and args.impl == "cmc":
        return run_ablation(args, torch.device("cuda", local))
    if args.impl == "reference":
        return run_reference(args, w, world, rank)
    return run_gpu(args, w, world, rank, local)


if __name__ == "__main__":
    sys.exit(main())
