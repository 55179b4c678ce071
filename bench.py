#!/usr/bin/env python
"""Benchmark of the NetKV scoring path on GB300.

Workload: 4,096 independent replicas of the single-stream 64-GPU cluster
(8 prefill + 8 decode instances at TP=4, 1,000 requests each, decode caches of
200K block hashes, indexed per replica as block hash -> decode mask), run as 4,096
concurrent streams whose
score weights cover a 16x16x16 grid.  One step is the whole hot path over all
streams: level bottlenecks of every telemetry snapshot (netkv_oracle_build),
prefix hits of every (request, decode) pair (netkv_prefix_match) and the greedy
of every stream (netkv_schedule_streams).  The decode caches are resident state
built once before timing (netkv_cache_build).

Prints one JSON line.  ``--impl reference`` times the CPU oracle instead, on a
bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "decisions/sec"
# the paper's compute-load model for --load-model: t_iter = 12 ms + 0.4 ms per batch slot
# (free constants: the paper's fit is not printed), 64 batch slots, 1 GB held back and
# 45 GB free per decode GPU at the start (Sec. VI-A); the same in the CPU oracle leg
LOAD_MODEL = (float(np.float32(0.012)), float(np.float32(0.0004)), 64, 0, 10 ** 9, 45 * 10 ** 9)
UNIT = "decisions/s"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="netkv", choices=["netkv", "reference"])
    ap.add_argument("--workload", default="replicas",
                    choices=["replicas", "single", "sweep", "longctx", "cluster"],
                    help="replicas: the 4,096-stream scoring step (default); single: one "
                         "stream of the 64-GPU cluster, its step and one decision replayed "
                         "from CUDA graphs (latency); sweep: the oracle-build sweep (1,000 "
                         "snapshots x 2,048 x 8,192 pairs); longctx, cluster: the long-"
                         "context and large-cluster steps")
    ap.add_argument("--keys", type=int, default=0,
                    help="cached blocks per decode (0 = the workload's own; smaller values give "
                         "reduced cases for ncu captures)")
    ap.add_argument("--requests", type=int, default=0,
                    help="requests per stream (0 = the workload's own; smaller values give "
                         "the reduced cases that ncu captures run on)")
    ap.add_argument("--snapshots", type=int, default=1000)
    ap.add_argument("--directed", action="store_true",
                    help="directed links: separate upward and downward utilisation rows")
    ap.add_argument("--load-model", action="store_true",
                    help="the paper's compute-load model (T_queue + T_decode, memory filter) "
                         "instead of the token load")
    ap.add_argument("--tiers", action="store_true",
                    help="the paper's per-tier maps: four congestion values per snapshot")
    ap.add_argument("--inflight", type=int, default=0,
                    help="self-contention counter cap (Eq. 4's n_inflight; the paper uses 16); "
                         "0 = the plain greedy")
    ap.add_argument("--evolving", type=int, default=0,
                    help="evolving LRU decode caches of this many blocks (the simulator's "
                         "caches, Sec. VI-B; 200000 = the configs' cache size); 0 = static "
                         "caches")
    ap.add_argument("--evolving-batch", type=int, default=1024,
                    help="streams whose caches are held at once (the state of a 200,000-block "
                         "cache is 12 MiB)")
    ap.add_argument("--streams", type=int, default=4096)
    ap.add_argument("--cpu-streams", type=int, default=256,
                    help="streams of the multi-core CPU-oracle sample (one per core at a time)")
    ap.add_argument("--cpu-streams-1t", type=int, default=12,
                    help="streams of the one-thread CPU-oracle sample")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--table-batch", type=int, default=256)
    ap.add_argument("--e2e-copy-chains", action="store_true",
                    help="e2e: copy the chains to the device instead of reading them in place")
    ap.add_argument("--no-fuse", action="store_true",
                    help="build the level bottlenecks UB in their own pass (netkv_oracle_build) "
                         "instead of from the utilisation rows inside the base-score pass")
    ap.add_argument("--no-share", action="store_true",
                    help="prefix match without the workspace (no grouping of shared prefixes)")
    return ap.parse_args()


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def rank_seed0(rank: int, streams: int) -> int:
    """Weak scaling: rank k runs its own replicas, seeds [k*streams, (k+1)*streams)."""
    return rank * streams


def max_over_ranks(x: float, device=None) -> float:
    """Maximum of a per-rank value over all ranks (the step time of the slowest rank)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def workload_config(streams, world, extra=None, kind="replicas"):
    if kind == "single":
        cfg = {"workload": "single stream, 64-GPU four-tier tree (8P+8D, TP=4), 1,000 "
                           "requests, decode caches of 200K blocks: the stream's whole step "
                           "and one decision, each replayed from a CUDA graph",
               "streams_per_gpu": 1, "requests_per_stream": 1000, "decodes": 8,
               "prefills": 8, "parallelism": f"replicas{world}",
               "l2": "L2 flushed between timed iterations (256 MiB written): the stream's "
                     "inputs fit in L2"}
    elif kind == "longctx":
        cfg = {"workload": "prefix-heavy long context: 1,280-instance 8-ary tree (256P+1,024D), "
                           "64 streams x 256 requests of 131,072 tokens (8,192-block chains) "
                           "over 8 shared roots, decode caches of 2^20 blocks, full R x D match",
               "streams_per_gpu": 64, "requests_per_stream": 256, "decodes": 1024,
               "prefills": 256, "parallelism": f"replicas{world}",
               "l2": "inputs larger than L2 (cache index 64 GiB + chains 1 GiB per GPU)"}
    elif kind == "cluster":
        cfg = {"workload": "large cluster: 5,120-instance 8-ary tree (1,024P+4,096D), "
                           "16 streams x 100,000 requests sharing caches of 200K blocks and "
                           "telemetry",
               "streams_per_gpu": 16, "requests_per_stream": 100_000, "decodes": 4096,
               "prefills": 1024, "parallelism": f"replicas{world}",
               "l2": "inputs larger than L2 (cache index 4 GiB, M 13 GB per GPU)"}
    else:
        cfg = {"workload": f"{streams} replicas x 64-GPU four-tier tree (8P+8D, TP=4), "
                           "1,000 requests/stream, decode caches of 200K blocks",
               "streams_per_gpu": streams, "requests_per_stream": 1000, "decodes": 8,
               "prefills": 8, "parallelism": f"replicas{world}",
               "l2": "inputs larger than L2 (cache index 100 GiB + chains 27 GB per GPU)"}
    if extra:
        cfg.update(extra)
    return cfg


# ------------------------------------------------------------------ clocks
class Clocks:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        # one more sample at the end of the timed region (still under load: the caller
        # stops the sampler before synchronising on the last launches' completion)
        try:
            with open(self.path, "a") as f:
                subprocess.run(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                "--format=csv,noheader,nounits"], stdout=f,
                               stderr=subprocess.DEVNULL, timeout=10)
        except (OSError, subprocess.TimeoutExpired):
            pass
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "samples": len(sm), "reasons": sorted(reasons)}


# The kernel code a call's DRAM traffic was measured on: source files, each up to an
# optional marker line (code after the marker, such as another entry point, does not
# change the call's kernels).
KERNEL_CODE = {
    "prefix_match": [("paper_2606_03910_gb300/csrc/prefix.cu", "// netkv_prefix_match_static:"),
                     ("paper_2606_03910_gb300/csrc/cache_index.cuh", None),
                     ("paper_2606_03910_gb300/csrc/netkv_internal.cuh", None)],
    "oracle_build": [("paper_2606_03910_gb300/csrc/oracle_build.cu", None),
                     ("paper_2606_03910_gb300/csrc/netkv_internal.cuh", None)],
}

# DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum over the call's kernels) from
# one-kernel ncu captures of a reduced case, per unit of work, keyed by the hash of the
# kernel code it was measured on; a changed kernel reports null until re-measured.
#   prefix_match: bytes per request, from the 64-replica case of the bench workload
#   oracle_build: bytes per snapshot of the oracle-build sweep
MEASURED_TRAFFIC = {
    # 64 replicas (64,000 requests): group_insert 8.96 MB, group_resolve 2.20 MB,
    # match_leaders 92.51 MB, match_members_kernel 239.84 MB (read + write)
    "prefix_match": {"code_sha256_16": "770ae3653abd8151", "bytes_per_unit": 343_515_136 / 64_000,
                     "unit": "request", "captured": "64-replica case, one launch per kernel"},
    "oracle_build": {"code_sha256_16": "ed437e71560780e2", "bytes_per_unit": 67_155_930,
                     "unit": "snapshot", "captured": "1,000-snapshot sweep, one launch"},
}


def kernel_code_hash(kernel: str):
    import hashlib
    h = hashlib.sha256()
    for path, marker in KERNEL_CODE[kernel]:
        try:
            with open(os.path.join(ROOT, path)) as f:
                text = f.read()
        except OSError:
            return None
        if marker is not None and marker in text:
            text = text[:text.index(marker)]
        h.update(path.encode())
        h.update(text.encode())
    return h.hexdigest()[:16]


def measured_traffic(kernel: str, units: int):
    """DRAM bytes of one launch of `kernel` over `units` units of work, or None when the
    kernel code changed since the measurement."""
    m = MEASURED_TRAFFIC.get(kernel)
    if not m or m["code_sha256_16"] is None or m["code_sha256_16"] != kernel_code_hash(kernel):
        return None
    return int(round(m["bytes_per_unit"] * units))


def sweep_traffic(n_snap: int):
    """oracle_build's traffic is one pass over the output, so it scales with the snapshots."""
    return measured_traffic("oracle_build", n_snap)


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


# ------------------------------------------------------------------ CPU oracle
def cpu_oracle_sample(w, streams, theta, cap, bpt, inflight=0, directed=False, tiers=False,
                      load_model=False, threads=None, omp_threads=1):
    """Time the CPU oracle alone on whole streams of the workload: its prefix match and its
    greedy (with self-contention when inflight > 0, directed links, per-tier maps or the
    compute-load model as asked).  The streams' inputs (key lists, chains, telemetry rows)
    are gathered from the generator before the clock starts.  threads = None: the streams
    run concurrently, one per host core at a time, each oracle call on one OpenMP thread;
    threads = 1: one after another on the calling thread, each oracle call on omp_threads
    OpenMP threads (the prefix match is parallel over a stream's requests).
    Returns (decisions, seconds, threads used)."""
    import concurrent.futures as cf
    import oracle
    from oracle.workload import solve_stream, stream_inputs
    with cf.ThreadPoolExecutor(cpu_cores()) as ex:  # generator output, before the clock
        xs = list(ex.map(lambda s: stream_inputs(w, int(s), directed=directed, tiers=tiers),
                         streams))
    lm = None
    if load_model:
        a, b, bmax, _, m_min, m0 = LOAD_MODEL
        lm = (a, b, bmax, m_min, m0)
    n_threads = cpu_cores() if threads is None else int(threads)
    oracle.lib()

    def solve(x):
        oracle.set_threads(omp_threads if n_threads == 1 else 1)
        _, res = solve_stream(w, x, theta, cap, bpt, inflight, lm, tiers)
        return int(res.dec.shape[0])

    if n_threads == 1:
        oracle.set_threads(omp_threads)
        t0 = time.perf_counter()
        dec = sum(solve(x) for x in xs)
        secs = time.perf_counter() - t0
        oracle.set_threads(cpu_cores())
    else:
        with cf.ThreadPoolExecutor(n_threads) as ex:
            t0 = time.perf_counter()
            dec = sum(ex.map(solve, xs))
            secs = time.perf_counter() - t0
    return dec, secs, min(n_threads, len(xs))


def cpu_baseline_line(w, n_streams, args, theta, cap, bpt, note=""):
    """cpu_baseline of a streamed workload: the oracle on a sample of whole streams across
    the host cores, and on a smaller sample with one thread."""
    rng = np.random.default_rng(0)
    sample = rng.choice(n_streams, size=min(args.cpu_streams, n_streams), replace=False)
    d, secs, used = cpu_oracle_sample(w, sample, theta, cap, bpt, args.inflight, args.directed,
                                      args.tiers, args.load_model)
    s1 = sample[:max(1, min(args.cpu_streams_1t, len(sample)))]
    d1, secs1, _ = cpu_oracle_sample(w, s1, theta, cap, bpt, args.inflight, args.directed,
                                     args.tiers, args.load_model, threads=1)
    return {"value": d / secs, "unit": UNIT, "cores": used, "kind": "oracle",
            "sample": f"{len(sample)} of {n_streams} whole streams ({d} decisions in "
                      f"{secs:.1f} s), prefix match + greedy, inputs generated before timing, "
                      f"one stream per core at a time{note}",
            "one_thread": {"value": d1 / secs1, "unit": UNIT, "cores": 1,
                           "sample": f"{len(s1)} whole streams ({d1} decisions in {secs1:.1f} s)"}}


def cpu_oracle_sample_large(w, s, n_req, n_dec, theta, cap, bpt):
    """Oracle time per decision on a workload whose caches are too large for the oracle's
    whole-stream sets: its matcher over the first n_req requests of stream s against
    n_dec evenly spaced decodes (time scaled by D / n_dec), plus its greedy over those
    requests' events given the generator's constructed hits.  Key and chain generation
    stay outside the timed parts.  Returns (decisions, seconds)."""
    import oracle
    import synth
    spec = w.spec
    r0 = int(w.req_off[s])
    r1 = min(int(w.req_off[s + 1]), r0 + n_req)
    g = int(synth.request_set(w)[r0])
    chains = w.chains(r0, r1)
    chain_off = (w.chain_off[r0:r1 + 1] - w.chain_off[r0]).astype(np.uint64)
    t_match = 0.0
    decs = np.unique(np.linspace(0, w.D - 1, n_dec).astype(np.int64))
    for d in decs:
        keys = w.keys(g, int(d))
        t0 = time.perf_counter()
        oracle.prefix_match_one(keys, chains, chain_off)
        t_match += time.perf_counter() - t0
    t_match *= w.D / len(decs)
    ev = w.events[int(w.event_off[s]):int(w.event_off[s + 1])].astype(np.uint64)
    rr = (ev & np.uint64(0x7FFFFFFF)).astype(np.int64)
    keep = rr < r1
    ev_local = ((rr[keep] - r0).astype(np.uint64) |
                (ev[keep] & np.uint64(1 << 31))).astype(np.uint32)
    snaps, snap_local = np.unique(w.snap[r0:r1].astype(np.int64), return_inverse=True)
    util = np.stack([w.util(int(k), int(k) + 1)[0] for k in snaps])
    M = synth.constructed_hits(w, r0, r1)
    wn, wp, wl = (float(v) for v in w.weights[s])
    t0 = time.perf_counter()
    oracle.schedule_stream(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, util,
                           w.length[r0:r1], w.prefill[r0:r1], snap_local.astype(np.uint32), M,
                           ev_local, wn, wp, wl, theta, cap, bpt)
    t_greedy = time.perf_counter() - t0
    return r1 - r0, t_match + t_greedy


def cpu_sweep_sample(spec, w, util, n_snap):
    """Time the CPU oracle building the full cost matrix of n_snap snapshots; returns
    (pair costs, seconds)."""
    import oracle
    t0 = time.perf_counter()
    C = oracle.cost_matrix(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, util[:n_snap],
                           spec.kv_bytes)
    return C.size, time.perf_counter() - t0


def cpu_cores():
    return int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))


# ------------------------------------------------------------------ reference arm
def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    if args.workload == "sweep":
        return run_reference_sweep(args, world)
    import synth
    if args.workload == "single":
        spec = synth.config0()
        n_streams = 1
    else:
        spec = synth.config1(args.streams)
        n_streams = args.streams
    if args.requests:
        spec.requests_per_stream = args.requests
    w = synth.make_workload(spec)
    theta = float(np.float32(synth.THETA_S_PER_TOKEN))
    per_step = 1
    order = np.random.default_rng(1).permutation(n_streams)
    k = 0
    # one whole stream per step; the oracle's prefix match runs on every host core
    # (OpenMP over the stream's requests), its greedy on one
    for _ in range(args.warmup):
        cpu_oracle_sample(w, order[k:k + per_step], theta, spec.cap_tokens,
                          synth.BYTES_PER_TOKEN_SHARD, args.inflight, threads=1,
                          omp_threads=cpu_cores())
        k = (k + per_step) % n_streams
    dec_total, secs = 0, 0.0
    for _ in range(args.steps):
        d, t, _ = cpu_oracle_sample(w, order[k:k + per_step], theta, spec.cap_tokens,
                                    synth.BYTES_PER_TOKEN_SHARD, args.inflight, threads=1,
                                    omp_threads=cpu_cores())
        dec_total += d
        secs += t
        k = (k + per_step) % n_streams
    value = dec_total / secs
    sample = (f"{per_step} whole stream per step (prefix match + greedy), inputs generated "
              "before timing")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * secs / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(args.streams, world, kind=args.workload),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cpu_cores(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def run_reference_sweep(args, world):
    import synth
    spec = synth.config3(args.snapshots)
    w = synth.make_workload(spec)
    util = w.util()
    for _ in range(args.warmup):
        cpu_sweep_sample(spec, w, util, 1)
    pairs, secs = 0, 0.0
    for _ in range(args.steps):
        n, t = cpu_sweep_sample(spec, w, util, 1)
        pairs += n
        secs += t
    value = pairs / secs
    line = {"impl": "reference", "metric": SWEEP_METRIC, "value": value, "unit": SWEEP_UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * secs / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": sweep_config(args.snapshots, spec, w),
            "cpu_baseline": {"value": value, "unit": SWEEP_UNIT, "cores": cpu_cores(),
                             "kind": "oracle",
                             "sample": "one snapshot's full cost matrix per step"},
            "e2e": {"value": value, "unit": SWEEP_UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def workload_spec(kind: str, streams: int, rank: int, requests: int = 0, keys: int = 0):
    """Generator spec of a bench workload; rank k takes its own seeds (weak scaling).
    requests > 0 sets the requests per stream, keys > 0 the cached blocks per decode
    (reduced cases)."""
    import synth
    if kind == "replicas":
        spec = synth.config1(streams)
        spec.seed0 = rank_seed0(rank, streams)
    elif kind == "single":
        spec = synth.config0()
        spec.seed0 = rank_seed0(rank, 1)
    elif kind == "longctx":
        spec = synth.config4()
        spec.seed0 = rank_seed0(rank, spec.n_streams)
    elif kind == "cluster":
        spec = synth.config2()
        spec.seed0 = rank_seed0(rank, spec.n_streams)
    else:
        raise ValueError(f"unknown workload {kind!r}")
    if requests:
        spec.requests_per_stream = int(requests)
    if keys:
        spec.n_keys = int(keys)
    return spec


def setup_workload(spec, dev, table_batch: int = 256, inflight: bool = False,
                   directed: bool = False, tiers: bool = False):
    """A generated workload on `dev`: its inputs, the resident cache index and the step's
    device buffers.  Returns (workload, scorer, step inputs, step outputs)."""
    import torch
    import synth
    import synth.device as sdev
    from synth import stage
    from paper_2606_03910_gb300 import netkv
    from paper_2606_03910_gb300.pipeline import Scorer, StepInputs, weights_tensor
    w = synth.make_workload(spec)
    theta = float(np.float32(synth.THETA_S_PER_TOKEN))
    bpt = synth.BYTES_PER_TOKEN_SHARD
    log2_index = netkv.index_log2_capacity(synth.distinct_keys_per_group(w))
    sc = Scorer(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, w.L, w.n_sets, log2_index,
                device=dev)
    for g0 in range(0, w.n_sets, table_batch):
        g1 = min(w.n_sets, g0 + table_batch)
        keys = sdev.keys(w, g0, g1, device=dev)
        sc.load_caches(keys, stage.key_offsets(w, (g1 - g0) * w.D, device=dev), set0=g0,
                       n_sets=g1 - g0)
        del keys
    torch.cuda.synchronize()
    if int(sc.status.item()) != 0:
        raise RuntimeError(f"cache build status {int(sc.status.item())}")
    ra = stage.request_arrays(w, device=dev)
    chains, _ = sdev.chains(w, device=dev)
    if tiers:  # the paper's per-tier maps: four congestion values per snapshot
        sc.oracle_mode = "tiers"
    util = stage.util(w, device=dev, direction="tiers") if tiers else sdev.util(w, device=dev)
    x = StepInputs(util=util, chains=chains, chain_off=ra["chain_off"],
                   set_off=ra["set_off"], length=ra["length"], prefill=ra["prefill"],
                   snap=ra["snap"], events=ra["events"], event_off=ra["event_off"],
                   weights=weights_tensor(w.weights, theta, spec.cap_tokens, bpt, device=dev),
                   arrival_us=(torch.from_numpy(w.arrival_us.astype(np.int64)).to(dev)
                               if inflight else None),
                   util_down=sdev.util(w, device=dev, direction="down") if directed else None)
    out = sc.alloc_outputs(x.n_snap, x.R, x.n_streams)
    return w, sc, x, out


def setup_replicas(streams: int, rank: int, dev, table_batch: int = 256):
    """The 4,096-replica workload (or `streams` replicas) of rank `rank` on `dev`."""
    return setup_workload(workload_spec("replicas", streams, rank), dev, table_batch)


def match_extent(M, chain_off, rows: int = 1 << 16):
    """(examined, probes) of a prefix-match result, in row chunks: blocks any exact matcher
    must examine (each chain up to the first miss of its last surviving decode, or its end)
    and per-(request, decode) probes up to each first miss."""
    import torch
    nblk_all = (chain_off[1:] - chain_off[:-1]).to(torch.int64)
    examined = probes = 0
    for r0 in range(0, M.shape[0], rows):
        m = M[r0:r0 + rows].to(torch.int32) & 0xFFFF
        nb = nblk_all[r0:r0 + rows]
        examined += int(torch.minimum(m.max(dim=1).values.to(torch.int64) + 1, nb).sum().item())
        probes += int(torch.minimum(m.to(torch.int64) + 1, nb[:, None]).sum().item())
    return examined, probes


# ------------------------------------------------------------------ GPU arm
def run_netkv(args):
    import torch
    import synth
    import __graft_entry__
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    __graft_entry__.build()
    from paper_2606_03910_gb300.pipeline import StepInputs

    w, sc, x, out = setup_workload(workload_spec(args.workload, args.streams, rank, args.requests,
                                                 args.keys), dev,
                                   args.table_batch, inflight=args.inflight > 0,
                                   directed=args.directed, tiers=args.tiers)
    sc.share_prefixes = not args.no_share
    sc.inflight_cap = args.inflight
    sc.fuse_level_bottlenecks = not args.no_fuse
    if args.load_model:
        from paper_2606_03910_gb300 import netkv
        sc.load_model = netkv.LoadModel(*LOAD_MODEL)
    theta = float(np.float32(synth.THETA_S_PER_TOKEN))
    bpt = synth.BYTES_PER_TOKEN_SHARD
    spec = w.spec
    stream = torch.cuda.current_stream(dev)
    for _ in range(args.warmup):
        sc.step(x, out, stream)
    torch.cuda.synchronize()
    if int(out.status.item()) != 0:
        raise RuntimeError(f"device status {int(out.status.item())} after warm-up")

    # ---- timed region: device-resident inputs
    fused = sc.fused(x)
    names = ("prefix_match", "schedule") if fused else ("oracle_build", "prefix_match", "schedule")
    calls = ((sc.prefix_match, sc.schedule) if fused
             else (sc.oracle_build, sc.prefix_match, sc.schedule))
    ev = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in names] for _ in range(args.steps)]
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = Clocks(local)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    t0.record(stream)
    for k in range(args.steps):
        for j, fn in enumerate(calls):
            ev[k][j][0].record(stream)
            fn(x, out, stream)
            ev[k][j][1].record(stream)
    t1.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    if world > 1:
        dist.barrier()
    ms = t0.elapsed_time(t1) / args.steps
    per_kernel = {n: sum(ev[k][j][0].elapsed_time(ev[k][j][1]) for k in range(args.steps)) / args.steps
                  for j, n in enumerate(names)}
    ms = max_over_ranks(ms, dev)
    status = int(out.status.item())
    if status != 0:
        raise RuntimeError(f"device status {status} in the timed region")

    R, D = x.R, sc.D
    # level bottlenecks 1; prefix match 4 (group insert, group resolve, leaders, members)
    # with a workspace or 1 without; greedy 2 (base scores + walk) with a workspace, 3 for
    # pools of 1,025 .. 4,096 decodes (base scores with chunk lists, list merge, listed
    # walk), or 1
    plain_greedy = not (sc.inflight_cap > 0 or sc.load_model is not None)
    listed = plain_greedy and sc.precompute_scores and 1025 <= sc.D <= 4096
    launches_per_step = (0 if fused else 1) + (4 if sc.share_prefixes else 1) + (
        1 if not plain_greedy else (3 if listed else 2) if sc.precompute_scores else 1)
    n_input_tensors = sum(1 for f in dataclasses.fields(StepInputs)
                          if isinstance(getattr(x, f.name), torch.Tensor))
    decisions = R * world
    value = decisions / (ms / 1e3)

    # ---- roofline of the dominant kernel (the prefix-match call)
    examined, probes = match_extent(out.M, x.chain_off)
    algo = {
        # floor: each chain block up to the request's last first miss read once (8 B) and
        # each M entry written once (2 B); index reads are left out (prefix sharing skips
        # them over shared prefixes and L2 serves most of the rest)
        "prefix_match": 8 * examined + 2 * R * D,
        # per snapshot: the utilisation row (L floats), 16-byte UB of every instance
        "oracle_build": 0 if fused else x.n_snap * (16 + 16 * sc.N) if args.tiers else
                        x.n_snap * ((8 if x.util_down is not None else 4) * w.L + 16 * sc.N),
        # per arrival: event, len/prefill/snap and the dec/best/second stores; per
        # departure: event, len, dec; the loads in and out.  With a workspace the base pass
        # reads M (2 B) and writes the base score (4 B) of every candidate, and the walk
        # reads the row (staged walk) or the candidate list and bound (listed walk: the
        # chunk lists written and merged, 264 B each); without one the walk reads M.
        "schedule": R * (4 + 12 + 12) + R * 12 + 2 * 8 * D * x.n_streams + (
            (R * 6 * D + (R * 264 * (2 * ((D + 1023) // 1024) + 2) if listed else R * 4 * D))
            if sc.precompute_scores else R * 2 * D),
    }
    dom = max(per_kernel, key=per_kernel.get)
    peak, peak_src = measured_peaks()
    achieved = algo[dom] / (per_kernel[dom] / 1e3) / 1e9
    traffic = None
    if dom == "prefix_match" and args.workload == "replicas":
        traffic = measured_traffic(dom, R)
    traffic_gbs = None if traffic is None else traffic / (per_kernel[dom] / 1e3) / 1e9
    roofline = {"kernel": dom, "bound": "hbm", "achieved": round(achieved, 1), "peak": peak,
                "unit": "GB/s", "frac": round(achieved / peak, 4),
                "traffic": traffic, "peak_source": peak_src,
                "traffic_achieved": None if traffic_gbs is None else round(traffic_gbs, 1),
                "traffic_frac": None if traffic_gbs is None else round(traffic_gbs / peak, 4),
                "traffic_source": (f"{MEASURED_TRAFFIC[dom]['captured']}, scaled by "
                                   f"{MEASURED_TRAFFIC[dom]['unit']}s" if traffic else None),
                "algorithmic_bytes_per_launch": algo[dom],
                "per_unit": {"prefix_match": "8 B per (request, chain block examined up to its "
                                             "last first miss) + 2 B per M entry",
                             "oracle_build": "per snapshot: the utilisation row + 16 B per instance",
                             "schedule": "per arrival: event, request fields, dec/best/second, "
                                         "M read and base score written per candidate (2 + 4 B), "
                                         "then the row (staged walk) or the 264 B candidate list "
                                         "(listed walk); per departure: event, len, dec"}[dom],
                "examined_blocks_per_launch": examined,
                "survey_probe_bytes_per_launch": 16 * probes + 2 * R * D,
                "survey_probes_per_launch": probes,
                "kernel_ms": {k: round(v, 4) for k, v in per_kernel.items()}}

    # ---- end to end through the public API with pinned host buffers
    e2e = None
    if not args.no_e2e:
        xh = StepInputs(**{f.name: (getattr(x, f.name).cpu().pin_memory()
                                    if isinstance(getattr(x, f.name), torch.Tensor) else None)
                           for f in dataclasses.fields(StepInputs)})
        res_h = {k: torch.empty_like(getattr(out, k), device="cpu").pin_memory()
                 for k in ("dec", "best", "second", "load_final")}
        zc = () if args.e2e_copy_chains else ("chains",)
        h2d = sum(int(t.numel() * t.element_size()) for f in dataclasses.fields(StepInputs)
                  if isinstance((t := getattr(xh, f.name)), torch.Tensor) and f.name not in zc)
        zc_bytes = sum(int(getattr(xh, n).numel() * getattr(xh, n).element_size()) for n in zc)
        d2h = sum(int(t.numel() * t.element_size()) for t in res_h.values())
        for _ in range(max(1, args.warmup)):
            sc.step_host(xh, x, out, res_h, stream, zero_copy=zc)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            sc.step_host(xh, x, out, res_h, stream, zero_copy=zc)
        e1.record(stream)
        torch.cuda.synchronize()
        ems = e0.elapsed_time(e1) / args.steps
        ems = max_over_ranks(ems, dev)
        if int(out.status.item()) != 0:
            raise RuntimeError(f"device status {int(out.status.item())} in the e2e region")
        if not (torch.equal(res_h["dec"], out.dec.cpu()) and torch.equal(res_h["best"], out.best.cpu())):
            raise RuntimeError("host-buffer step results differ from the device step")
        e2e = {"value": decisions / (ems / 1e3), "unit": UNIT, "ms_per_step": round(ems, 3),
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "host_read_in_place_bytes": zc_bytes,
               "host_read_in_place": list(zc),
               "gpu_launches_per_step": launches_per_step + n_input_tensors - len(zc) + 4}

    # ---- CPU oracle baseline, rank 0 at N=1 only
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu and args.workload == "replicas":
        cpu = cpu_baseline_line(w, x.n_streams, args, theta, spec.cap_tokens, bpt)
    elif rank == 0 and world == 1 and not args.no_cpu:
        n_req, n_dec = (256, 16) if args.workload == "longctx" else (2000, 32)
        d, secs = cpu_oracle_sample_large(w, 0, n_req, n_dec, theta, spec.cap_tokens, bpt)
        cpu = {"value": d / secs, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
               "sample": f"first {d} requests of stream 0: the oracle's matcher on {n_dec} "
                         f"of {w.D} decodes scaled to all, plus its greedy given the "
                         f"constructed hits ({secs:.1f} s)"}

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 4),
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": "f32", "data": "synthetic",
                "config": workload_config(args.streams, world, kind=args.workload,
                                          extra=dict(([("inflight_cap", args.inflight)]
                                                      if args.inflight else []) +
                                                     ([("links", "directed")]
                                                      if args.directed else []) +
                                                     ([("oracle", "per-tier maps")]
                                                      if args.tiers else []) +
                                                     ([("load", "queue/decode-step model")]
                                                      if args.load_model else [])) or None),
                "scores_per_s": value * D, "gpu_launches": launches_per_step * args.steps,
                "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "clocks": clk}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def one_decision_inputs(x, r: int, stream_index: int = 0):
    """Step inputs of a single arrival: request r of the stream with its own telemetry row,
    chain, weights and an event list of that arrival alone (the loads start at zero)."""
    import torch
    from paper_2606_03910_gb300.pipeline import StepInputs
    dev = x.length.device
    k = int(x.snap[r].item())
    c0, c1 = int(x.chain_off[r].item()), int(x.chain_off[r + 1].item())
    i32 = lambda v: torch.tensor(v, dtype=torch.int32, device=dev)
    i64 = lambda v: torch.tensor(v, dtype=torch.int64, device=dev)
    return StepInputs(util=x.util[k:k + 1].clone(), chains=x.chains[c0:c1].clone(),
                      chain_off=i64([0, c1 - c0]), set_off=i32([0, 1]),
                      length=x.length[r:r + 1].clone(), prefill=x.prefill[r:r + 1].clone(),
                      snap=i32([0]), events=i32([0]), event_off=i64([0, 1]),
                      weights=x.weights[32 * stream_index:32 * (stream_index + 1)].clone())


def run_single(args):
    """The single-stream workload (64-GPU cluster, 1,000 requests): the stream's whole
    step (level bottlenecks, prefix match, greedy) and one decision (the same three calls
    for one arrival), each captured once in a CUDA graph and replayed, with L2 flushed
    between timed replays."""
    import torch
    import synth
    import __graft_entry__
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    __graft_entry__.build()
    from paper_2606_03910_gb300.pipeline import StepInputs
    spec = workload_spec("single", 1, rank, args.requests)
    w, sc, x, out = setup_workload(spec, dev, 1)
    theta = float(np.float32(synth.THETA_S_PER_TOKEN))
    bpt = synth.BYTES_PER_TOKEN_SHARD
    R, D = x.R, sc.D
    sc.fuse_level_bottlenecks = not args.no_fuse
    stream = torch.cuda.Stream(dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)

    def capture(fn, share, precompute):
        sc.share_prefixes, sc.precompute_scores = share, precompute
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            for _ in range(max(3, args.warmup)):
                fn(stream)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn(stream)
        torch.cuda.synchronize()
        return g

    # the stream's step: grouping, leaders and members (with the workspace), base scores
    # (level bottlenecks from the utilisation rows) and the walk: 6 launches
    g_step = capture(lambda st: sc.step(x, out, st), True, True)
    step_launches = 6 if sc.fused(x) else 7
    # one decision: one request against the 8 decodes, no workspaces: 3 launches
    r_one = int(w.req_off[0]) + R // 2
    x1 = one_decision_inputs(x, r_one)
    o1 = sc.alloc_outputs(1, 1, 1)
    g_one = capture(lambda st: sc.step(x1, o1, st), False, False)

    def time_graph(g, steps):
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(steps)]
        with torch.cuda.stream(stream):
            for k in range(steps):
                flush.zero_()  # between timed replays: L2 holds none of the inputs
                ev[k][0].record(stream)
                g.replay()
                ev[k][1].record(stream)
        torch.cuda.synchronize()
        t = sorted(a.elapsed_time(b) for a, b in ev)
        return sum(t) / len(t), t[len(t) // 2]

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            g_step.replay()
            g_one.replay()
    torch.cuda.synchronize()
    clocks = Clocks(local)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    step_ms, step_med = time_graph(g_step, args.steps)
    one_ms, one_med = time_graph(g_one, args.steps)
    clk = clocks.stop()
    ms = max_over_ranks(step_ms, dev)
    for o in (out, o1):
        if int(o.status.item()) != 0:
            raise RuntimeError(f"device status {int(o.status.item())}")
    value = R * world / (ms / 1e3)

    # e2e: the step through the public API from pinned host buffers, results read back
    e2e = None
    if not args.no_e2e:
        sc.share_prefixes, sc.precompute_scores = True, True
        xh = StepInputs(**{f.name: (getattr(x, f.name).cpu().pin_memory()
                                    if isinstance(getattr(x, f.name), torch.Tensor) else None)
                           for f in dataclasses.fields(StepInputs)})
        res_h = {k: torch.empty_like(getattr(out, k), device="cpu").pin_memory()
                 for k in ("dec", "best", "second", "load_final")}
        h2d = sum(int(t.numel() * t.element_size()) for f in dataclasses.fields(StepInputs)
                  if isinstance((t := getattr(xh, f.name)), torch.Tensor))
        d2h = sum(int(t.numel() * t.element_size()) for t in res_h.values())
        with torch.cuda.stream(stream):
            for _ in range(max(1, args.warmup)):
                sc.step_host(xh, x, out, res_h, stream)
        torch.cuda.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(args.steps)]
        with torch.cuda.stream(stream):
            for k in range(args.steps):
                flush.zero_()
                ev[k][0].record(stream)
                sc.step_host(xh, x, out, res_h, stream)
                ev[k][1].record(stream)
        torch.cuda.synchronize()
        ems = max_over_ranks(sum(a.elapsed_time(b) for a, b in ev) / args.steps, dev)
        if not torch.equal(res_h["dec"], out.dec.cpu()):
            raise RuntimeError("host-buffer step results differ from the device step")
        e2e = {"value": R * world / (ems / 1e3), "unit": UNIT, "ms_per_step": round(ems, 4),
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "note": "eager launches (no graph): the step's inputs copied from pinned host "
                       "memory and its results read back every step"}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        d, secs, _ = cpu_oracle_sample(w, [0], theta, spec.cap_tokens, bpt, threads=1,
                                       omp_threads=cpu_cores())
        d1, secs1, _ = cpu_oracle_sample(w, [0], theta, spec.cap_tokens, bpt, threads=1)
        cpu = {"value": d / secs, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
               "sample": f"the whole stream ({d} decisions in {secs:.2f} s): prefix match on "
                         "every core (OpenMP over requests), greedy on one; inputs generated "
                         "before timing",
               "one_thread": {"value": d1 / secs1, "unit": UNIT, "cores": 1,
                              "sample": f"the whole stream ({secs1:.2f} s)"}}
    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 4),
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": "f32", "data": "synthetic",
                "config": workload_config(1, world, kind="single"),
                "scores_per_s": value * D, "gpu_launches": (step_launches + 3) * args.steps,
                "latency": {"stream_step_ms": round(step_ms, 4),
                            "stream_step_ms_median": round(step_med, 4),
                            "per_decision_us_amortised": round(1e3 * step_ms / R, 3),
                            "one_decision_ms": round(one_ms, 4),
                            "one_decision_ms_median": round(one_med, 4),
                            "launches": {"stream_step": step_launches, "one_decision": 3},
                            "paper": "decision latency below 1.5 ms at up to 1,024 GPUs "
                                     "(Sec. VI-I, Experiment 7), candidate pool of at most 12 "
                                     "after memory filtering (Sec. V-B); the paper's scheduler "
                                     "host is not stated"},
                "roofline": {"kernel": "stream step", "bound": "latency", "achieved": None,
                             "peak": None, "unit": None, "frac": None, "traffic": None,
                             "note": "one stream of 1,000 arrivals x 8 decodes moves about "
                                     "8 MB: launch- and dependency-bound, so no HBM "
                                     "roofline; the replicas workload carries it"},
                "cpu_baseline": cpu, "e2e": e2e, "clocks": clk}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def run_evolving(args):
    """The replicas workload with evolving LRU caches: one step is the level bottlenecks
    of every snapshot, then, per batch of streams, their caches set from the key lists
    (netkv_lru_init) and hits plus greedy in one walk (netkv_schedule_streams_evolving)."""
    import torch
    import synth
    import synth.device as sdev
    from synth import stage
    import __graft_entry__
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    __graft_entry__.build()
    from paper_2606_03910_gb300 import netkv
    from paper_2606_03910_gb300.pipeline import Scorer, StepInputs, weights_tensor
    spec = workload_spec("replicas", args.streams, rank, args.requests)
    w = synth.make_workload(spec)
    theta = float(np.float32(synth.THETA_S_PER_TOKEN))
    bpt = synth.BYTES_PER_TOKEN_SHARD
    sc = Scorer(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, w.L, w.n_sets, 1, device=dev,
                index=False)
    S, D = w.n_streams, sc.D
    batch = max(1, min(args.evolving_batch, S))
    sc.lru_setup(batch, args.evolving)
    keys = sdev.keys(w, 0, w.n_sets, device=dev)       # every stream's initial caches
    key_off = stage.key_offsets(w, w.n_sets * D, device=dev)
    ra = stage.request_arrays(w, device=dev)
    chains, _ = sdev.chains(w, device=dev)
    x = StepInputs(util=sdev.util(w, device=dev), chains=chains, chain_off=ra["chain_off"],
                   set_off=ra["set_off"], length=ra["length"], prefill=ra["prefill"],
                   snap=ra["snap"], events=ra["events"], event_off=ra["event_off"],
                   weights=weights_tensor(w.weights, theta, spec.cap_tokens, bpt, device=dev))
    out = sc.alloc_outputs(x.n_snap, x.R, x.n_streams)
    stream = torch.cuda.current_stream(dev)
    batches = [(j0, min(S, j0 + batch)) for j0 in range(0, S, batch)]

    def step(ev=None):
        if ev:
            ev[0].record(stream)
        sc.oracle_build(x, out, stream)
        if ev:
            ev[1].record(stream)
        for k, (j0, j1) in enumerate(batches):
            netkv.netkv_lru_init(sc.lru_state, (j1 - j0) * D, sc.lru_cfg, keys, key_off[j0 * D:],
                                 out.status, stream)
            if ev:
                ev[2 + 2 * k].record(stream)
            sc.schedule_evolving(x, out, stream, streams=(j0, j1))
            if ev:
                ev[3 + 2 * k].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if int(out.status.item()) != 0:
        raise RuntimeError(f"device status {int(out.status.item())} after warm-up")
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2 + 2 * len(batches))]
           for _ in range(args.steps)]
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = Clocks(local)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    t0.record(stream)
    for k in range(args.steps):
        step(evs[k])
    t1.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    ms = max_over_ranks(t0.elapsed_time(t1) / args.steps, dev)
    if int(out.status.item()) != 0:
        raise RuntimeError(f"device status {int(out.status.item())} in the timed region")
    nb = len(batches)
    t_build = sum(e[0].elapsed_time(e[1]) for e in evs) / args.steps
    t_init = sum(sum((e[1] if b == 0 else e[1 + 2 * b]).elapsed_time(e[2 + 2 * b]) for b in range(nb))
                 for e in evs) / args.steps
    t_walk = sum(sum(e[2 + 2 * b].elapsed_time(e[3 + 2 * b]) for b in range(nb))
                 for e in evs) / args.steps
    R = x.R
    value = R * world / (ms / 1e3)
    # algorithmic bytes of the walk: per (arrival, decode) probe up to the first miss a chain
    # block (8 B) and a table slot (16 B); per block a dispatch uses, its log entry (8 B) and
    # slot (16 B); per evicted block, as many again (taken as the blocks a dispatch adds
    # beyond its hits on the chosen decode)
    M = out.M.to(torch.int64) & 0xFFFF
    nblk = (x.chain_off[1:] - x.chain_off[:-1]).to(torch.int64)
    probes = int(torch.minimum(M + 1, nblk[:, None]).sum().item())
    dsel = out.dec.to(torch.int64)
    ok = dsel >= 0
    used = int(nblk[ok].sum().item())
    hits_sel = int(M[ok].gather(1, dsel[ok][:, None]).sum().item())
    algo = 24 * probes + 24 * used + 24 * max(0, used - hits_sel)
    peak, peak_src = measured_peaks()
    achieved = algo / (t_walk / 1e3) / 1e9
    roofline = {"kernel": "evolving_kernel (netkv_schedule_streams_evolving)", "bound": "hbm",
                "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4), "traffic": None, "peak_source": peak_src,
                "algorithmic_bytes_per_launch": algo,
                "per_unit": "24 B per (arrival, decode) probe up to the first miss, 24 B per "
                            "block used by a dispatch, 24 B per block it adds (evictions)",
                "note": "a sequential walk per stream: bound by each arrival's chain of "
                        "dependent probes, not by bandwidth",
                "kernel_ms": {"oracle_build": round(t_build, 4), "lru_init": round(t_init, 4),
                              "evolving_walk": round(t_walk, 4)}}
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        from oracle.workload import run_stream_evolving
        import concurrent.futures as cf
        import oracle
        sample = np.random.default_rng(0).choice(S, size=min(args.cpu_streams_1t, S),
                                                 replace=False)
        oracle.lib()

        def one(s):
            oracle.set_threads(1)
            t = time.perf_counter()
            res = run_stream_evolving(w, int(s), theta, spec.cap_tokens, bpt, args.evolving)
            return int(res.dec.shape[0]), time.perf_counter() - t

        with cf.ThreadPoolExecutor(cpu_cores()) as ex:
            t0w = time.perf_counter()
            got = list(ex.map(one, sample))
            wall = time.perf_counter() - t0w
        d = sum(g[0] for g in got)
        cpu = {"value": d / wall, "unit": UNIT, "cores": min(cpu_cores(), len(sample)),
               "kind": "oracle",
               "sample": f"{len(sample)} whole streams ({d} decisions in {wall:.1f} s), one per "
                         "core; each includes gathering its key lists and chains from the "
                         "generator (about a tenth of its time)",
               "one_thread": {"value": d / sum(g[1] for g in got), "unit": UNIT, "cores": 1,
                              "sample": "the same streams, per-thread time"}}
    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 4),
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": "f32", "data": "synthetic",
                "config": workload_config(args.streams, world, kind="replicas",
                                          extra={"caches": f"evolving, LRU of {args.evolving} "
                                                           "blocks per decode (Sec. VI-B)",
                                                 "streams_per_batch": batch}),
                "scores_per_s": value * D, "gpu_launches": (1 + 2 * nb) * args.steps,
                "roofline": roofline, "cpu_baseline": cpu, "e2e": None, "clocks": clk}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


SWEEP_METRIC = "pair-costs/sec"
SWEEP_UNIT = "pair-costs/s"


def sweep_config(S, spec, w):
    P = int((w.role == 0).sum())
    D = int((w.role == 1).sum())
    return {"workload": f"oracle-build sweep: {S} snapshots x {P} x {D} pairs, "
                        f"{w.L}-link rows, Beta(2,5) + 5% hot links, KV {spec.kv_bytes / 1e9:g} GB",
            "l2": f"output {4 * S * P * D / 1e9:.1f} GB per step, larger than L2"}


def run_sweep(args):
    """Oracle-build sweep: the full fp32 C[s][p][d] rebuilt for every telemetry snapshot."""
    import torch
    import synth
    import __graft_entry__
    from paper_2606_03910_gb300 import netkv
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    __graft_entry__.build()
    spec = synth.config3(args.snapshots)
    spec.seed0 = rank
    w = synth.make_workload(spec)
    util_h = w.util()
    util = torch.from_numpy(util_h).to(dev)
    topo = netkv.netkv_topology_create(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, w.L)
    _, P, D, _ = netkv.netkv_topology_query(topo)
    S = args.snapshots
    C = torch.empty((S, P, D), dtype=torch.float32, device=dev)
    st = torch.zeros(1, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)
    for _ in range(args.warmup):
        netkv.netkv_oracle_build(topo, util, S, spec.kv_bytes, C, None, st, stream)
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = Clocks(local)
    clocks.start()
    t0.record(stream)
    for _ in range(args.steps):
        netkv.netkv_oracle_build(topo, util, S, spec.kv_bytes, C, None, st, stream)
    t1.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    ms = max_over_ranks(t0.elapsed_time(t1) / args.steps, dev)
    if int(st.item()) != 0:
        raise RuntimeError(f"device status {int(st.item())}")
    pairs = S * P * D
    peak, src = measured_peaks()
    algo = 4 * pairs + S * w.L * 4
    achieved = algo / (ms / 1e3) / 1e9
    e2e = None
    if not args.no_e2e:
        # each step takes the snapshots' utilisation rows from pinned host memory, rebuilds
        # C on the device (where the greedy reads it) and reads the status word back
        util_p = torch.from_numpy(util_h).pin_memory()
        st_p = torch.zeros(1, dtype=torch.int32).pin_memory()
        ub = util_p.numel() * 4
        for _ in range(args.warmup):
            netkv.netkv_copy_async(util, util_p, ub, stream)
            netkv.netkv_oracle_build(topo, util, S, spec.kv_bytes, C, None, st, stream)
            netkv.netkv_copy_async(st_p, st, 4, stream)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            netkv.netkv_copy_async(util, util_p, ub, stream)
            netkv.netkv_oracle_build(topo, util, S, spec.kv_bytes, C, None, st, stream)
            netkv.netkv_copy_async(st_p, st, 4, stream)
        e1.record(stream)
        torch.cuda.synchronize()
        if int(st_p.item()) != 0:
            raise RuntimeError(f"device status {int(st_p.item())}")
        ems = max_over_ranks(e0.elapsed_time(e1) / args.steps, dev)
        e2e = {"value": pairs * world / (ems / 1e3), "unit": SWEEP_UNIT,
               "ms_per_step": round(ems, 3), "h2d_bytes_per_step": ub, "d2h_bytes_per_step": 4}
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        n, t = cpu_sweep_sample(spec, w, util_h, 8)
        cpu = {"value": n / t, "unit": SWEEP_UNIT, "cores": cpu_cores(), "kind": "oracle",
               "sample": "the full cost matrix of the first 8 snapshots"}
    line = {"metric": SWEEP_METRIC, "value": pairs * world / (ms / 1e3), "unit": SWEEP_UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(ms, 4), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": sweep_config(S, spec, w),
            "gpu_launches": args.steps, "e2e": e2e,
            "roofline": {"kernel": "oracle_build", "bound": "hbm", "achieved": round(achieved, 1),
                         "peak": peak, "unit": "GB/s", "frac": round(achieved / peak, 4),
                         "traffic": sweep_traffic(S), "peak_source": src,
                         "algorithmic_bytes_per_launch": algo,
                         "per_unit": "4 B per pair written + the utilisation rows read"},
            "cpu_baseline": cpu, "clocks": clk}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def main():
    args = parse()
    if (args.inflight > 0) + args.directed + args.tiers + args.load_model + (args.evolving > 0) > 1:
        raise SystemExit("--inflight, --directed, --tiers, --load-model and --evolving are "
                         "measured one at a time")
    if args.evolving and args.workload != "replicas":
        raise SystemExit("--evolving runs on the replicas workload (one table set per stream)")
    if args.impl == "reference":
        return run_reference(args)
    if args.workload == "sweep":
        return run_sweep(args)
    if args.workload == "single":
        return run_single(args)
    if args.evolving:
        return run_evolving(args)
    return run_netkv(args)


if __name__ == "__main__":
    sys.exit(main())
