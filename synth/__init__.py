"""Seeded synthetic workload generators for NetKV decode-instance scoring.

This module is shared by the CUDA path and the CPU oracle: it produces input
arrays only (topologies, telemetry snapshots, request traces, block-hash
chains, cache contents, event lists, weights) and contains none of the
method's arithmetic (no tiers, paths, bottlenecks, prefix matching or scores).

Every random value is a pure function of (seed, purpose, index...) through
SplitMix64's output function (Steele, Lea and Flood, "Fast splittable
pseudorandom number generators", OOPSLA 2014), so any element can be produced
on its own: the host (numpy, here) and the device (``synth/synth_dev.cu``)
implement the same integer definitions and produce identical bytes for
chains, cache keys and uniform utilisations.  Values that need a logarithm
(lognormal lengths, Poisson gaps, Beta utilisations) are made on the host
only and copied to whichever side needs them.

Workload shapes follow the paper's evaluation setup (Sec. VI-A): Llama-3-70B
at TP=4 (Sec. III-B, Eq. 1), 16-token blocks, a four-tier tree of instances,
per-link utilisation snapshots refreshed every 100 ms and read 50 ms stale.
The paper's traces are not available; these synthetic inputs stand in for
them.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Tuple

import numpy as np

U64 = np.uint64
GOLDEN = 0x9E3779B97F4A7C15
MIX1 = 0xBF58476D1CE4E5B9
MIX2 = 0x94D049BB133111EB
MASK64 = (1 << 64) - 1

# purpose tags (one independent stream of draws per purpose)
P_LEN, P_OUT, P_GAP, P_PREFILL, P_ROOT, P_SHARE = 1, 2, 3, 4, 5, 6
P_ROOTHASH, P_TAIL, P_FILLER, P_DEPTH, P_UTIL, P_HOTSEL, P_HOT, P_BETA = (
    7, 8, 9, 10, 11, 12, 13, 14)

BLOCK_TOKENS = 16                      # B_tok, Sec. III-B
KV_BYTES_PER_TOKEN = 2 * 80 * 8 * 128 * 2   # Llama-3-70B fp16, Eq. 1
TP = 4
BYTES_PER_TOKEN_SHARD = KV_BYTES_PER_TOKEN // TP
HBM_FREE_BYTES = 45e9                  # free HBM per GPU, Sec. VI-A
CAP_TOKENS = int(HBM_FREE_BYTES // BYTES_PER_TOKEN_SHARD)   # 549,316
THETA_S_PER_TOKEN = 1e-6
TBT_US = 13_000                        # ~13 ms per output token (absolute TBT), Sec. VI-J
SNAP_PERIOD_US = 100_000
SNAP_STALE_US = 50_000
EMPTY_HASH_REMAP = GOLDEN              # hash value 0 is reserved as "empty"


# --------------------------------------------------------------------------
# counter-based generator
# --------------------------------------------------------------------------
def _mix_int(z: int) -> int:
    z &= MASK64
    z = ((z ^ (z >> 30)) * MIX1) & MASK64
    z = ((z ^ (z >> 27)) * MIX2) & MASK64
    return z ^ (z >> 31)


def _mix(z: np.ndarray) -> np.ndarray:
    with np.errstate(over="ignore"):
        z = (z ^ (z >> U64(30))) * U64(MIX1)
        z = (z ^ (z >> U64(27))) * U64(MIX2)
        return z ^ (z >> U64(31))


def stream_key(seed: int, purpose: int) -> int:
    return _mix_int((seed * GOLDEN + purpose) & MASK64)


def draw(seed: int, purpose: int, a, b=0) -> np.ndarray:
    """u64 draw for (seed, purpose, a, b); a and b broadcast as arrays."""
    k = U64(stream_key(seed, purpose))
    a = np.asarray(a, dtype=U64)
    b = np.asarray(b, dtype=U64)
    with np.errstate(over="ignore"):
        k2 = _mix(k + (a + U64(1)) * U64(GOLDEN))
        return _mix(k2 + (b + U64(1)) * U64(GOLDEN))


def unit(x: np.ndarray) -> np.ndarray:
    """u64 -> double uniform in [0, 1) from the top 53 bits."""
    return (x >> U64(11)).astype(np.float64) * (1.0 / 9007199254740992.0)


def below(x: np.ndarray, n) -> np.ndarray:
    """u64 -> integer uniform in [0, n) by the multiply-high rule on 32 bits."""
    n = np.asarray(n, dtype=U64)
    return ((x >> U64(32)) * n) >> U64(32)


def nonzero_hash(x: np.ndarray) -> np.ndarray:
    return np.where(x == U64(0), U64(EMPTY_HASH_REMAP), x)


def uniform09_f32(x: np.ndarray) -> np.ndarray:
    """u64 -> fp32 utilisation in [0, 0.9): an integer m < 0.9*2^24 scaled by 2^-24 (exact)."""
    m = ((x >> U64(40)) * U64(9)) // U64(10)
    return (m.astype(np.float32) * np.float32(2.0 ** -24)).astype(np.float32)


def lognormal(seed: int, purpose: int, idx: np.ndarray, median: float, sigma: float) -> np.ndarray:
    u1 = unit(draw(seed, purpose, idx, 0))
    u2 = unit(draw(seed, purpose, idx, 1))
    z = np.sqrt(-2.0 * np.log1p(-u1)) * np.cos(2.0 * np.pi * u2)
    return median * np.exp(sigma * z)


# --------------------------------------------------------------------------
# workload specification
# --------------------------------------------------------------------------
@dataclasses.dataclass
class Spec:
    name: str
    fanout: Tuple[int, int, int, int]           # instances/node, nodes/leaf, leaves/pod, pods
    role_rule: str                              # "segregated" | "mod5" | "alternate"
    tier_bw: Tuple[float, float, float, float] = (900e9, 400e9, 200e9, 100e9)   # B/s
    tier_lat: Tuple[float, float, float, float] = (1e-6, 3e-6, 6e-6, 10e-6)     # s
    n_links: Optional[int] = None               # utilisation vector length (>= used edges)
    n_streams: int = 1
    requests_per_stream: int = 1000
    rate_per_s: float = 5.0
    len_mode: str = "lognormal"                 # "lognormal" | "fixed"
    len_median: float = 8192.0
    len_sigma: float = 1.0
    len_clip: Tuple[int, int] = (512, 131072)
    len_fixed: int = 131072
    n_roots: int = 50
    root_blocks: Tuple[int, ...] = (8192,)      # one value for all roots, or one per root
    share_mode: str = "frac"                    # "frac": floor(U[0,0.9]*n); "root": whole root
    n_keys: int = 200_000
    log2_cap: int = 19
    depth_mode: str = "scaled"                  # "scaled" | "uniform"
    util_mode: str = "uniform09"                # "uniform09" | "beta25_hot"
    n_snapshots: Optional[int] = None           # fixed snapshot count (oracle sweep)
    tables: str = "per_stream"                  # "per_stream" | "shared"
    telemetry: str = "per_stream"               # "per_stream" | "shared"
    weights: str = "unit"                       # "unit" | "grid16"
    seed0: int = 0
    kv_bytes: float = 10e9                      # oracle-build sweep payload
    cap_tokens: int = CAP_TOKENS

    def root_len(self, k: np.ndarray) -> np.ndarray:
        rb = np.asarray(self.root_blocks, dtype=np.int64)
        return rb[np.minimum(k, len(rb) - 1)] if len(rb) > 1 else np.full(np.shape(k), rb[0], np.int64)


def config0() -> Spec:
    """Single stream, 64-GPU four-tier tree at TP=4: 8 prefill + 8 decode instances."""
    return Spec(name="single-stream-64gpu", fanout=(1, 2, 2, 4), role_rule="segregated")


def config1(n_streams: int = 4096) -> Spec:
    """4,096 independent replicas of the single-stream workload (seed and weights vary)."""
    return Spec(name="replicas-4096x64gpu", fanout=(1, 2, 2, 4), role_rule="segregated",
                n_streams=n_streams, weights="grid16")


def config2(n_streams: int = 16, requests_per_stream: int = 100_000) -> Spec:
    """8-ary four-tier tree, 1,024 prefill + 4,096 decode instances, 16 streams of 100K requests."""
    return Spec(name="large-cluster-5120", fanout=(1, 8, 8, 80), role_rule="mod5",
                n_streams=n_streams, requests_per_stream=requests_per_stream,
                rate_per_s=400.0, tables="shared", telemetry="shared")


def config3(n_snapshots: int = 1000) -> Spec:
    """Oracle-build sweep: 2,048 x 8,192 pairs, 24,576-link snapshots, Beta(2,5) + 5% hot links."""
    return Spec(name="oracle-sweep-2048x8192", fanout=(1, 8, 8, 160), role_rule="mod5",
                n_links=24_576, n_streams=0, util_mode="beta25_hot",
                n_snapshots=n_snapshots, telemetry="shared", kv_bytes=10e9)


def config4_root_blocks() -> Tuple[int, ...]:
    return tuple(int(round(256 + k * (7680 - 256) / 7)) for k in range(8))


def config4(n_streams: int = 64, requests_per_stream: int = 256) -> Spec:
    """Prefix-heavy long context: 1,024 decode tables of 2^20 keys at load factor 0.5."""
    return Spec(name="prefix-heavy-1024x16384", fanout=(1, 8, 8, 20), role_rule="mod5",
                n_streams=n_streams, requests_per_stream=requests_per_stream,
                len_mode="fixed", len_fixed=131072, n_roots=8,
                root_blocks=config4_root_blocks(), share_mode="root",
                n_keys=1 << 20, log2_cap=21, depth_mode="uniform",
                tables="shared", telemetry="shared")


CONFIGS = {0: config0, 1: config1, 2: config2, 3: config3, 4: config4}


# --------------------------------------------------------------------------
# topology inputs (roles only; no tiers or paths here)
# --------------------------------------------------------------------------
def roles(spec: Spec) -> np.ndarray:
    f0, f1, f2, f3 = spec.fanout
    n = f0 * f1 * f2 * f3
    i = np.arange(n)
    if spec.role_rule == "segregated":
        # per pod: first half of the leaves prefill, second half decode
        leaf_in_pod = (i // (f0 * f1)) % f2
        return (leaf_in_pod >= f2 // 2).astype(np.uint8)
    if spec.role_rule == "mod5":
        return (i % 5 != 0).astype(np.uint8)
    if spec.role_rule == "alternate":
        return (i % 2 == 1).astype(np.uint8)
    raise ValueError(spec.role_rule)


def used_links(spec: Spec) -> int:
    f0, f1, f2, f3 = spec.fanout
    n = f0 * f1 * f2 * f3
    return n + f1 * f2 * f3 + f2 * f3 + f3


def n_links(spec: Spec) -> int:
    return spec.n_links if spec.n_links is not None else used_links(spec)


# --------------------------------------------------------------------------
# workload
# --------------------------------------------------------------------------
@dataclasses.dataclass
class Workload:
    spec: Spec
    role: np.ndarray            # u8 [N]
    P: int
    D: int
    L: int                      # utilisation vector length
    # requests (global index r; streams are contiguous ranges)
    req_off: np.ndarray         # i64 [n_streams+1]
    stream_seed: np.ndarray     # i64 [n_streams]
    length: np.ndarray          # u32 [R] tokens
    prefill: np.ndarray         # u32 [R] prefill rank
    arrival_us: np.ndarray      # i64 [R]
    depart_us: np.ndarray       # i64 [R]
    snap: np.ndarray            # u32 [R] global snapshot index
    root: np.ndarray            # u32 [R]
    shared: np.ndarray          # u32 [R] leading root blocks
    chain_off: np.ndarray       # u64 [R+1]
    # caches
    n_sets: int
    set_off: np.ndarray         # u32 [n_sets+1] request ranges per table set
    set_seed: np.ndarray        # i64 [n_sets]
    depth: np.ndarray           # i64 [n_sets, D, n_roots]
    # telemetry
    n_snap: int
    snap_seed: np.ndarray       # i64 [n_snap] telemetry seed of each snapshot
    snap_local: np.ndarray      # i64 [n_snap] snapshot index within its telemetry stream
    # events
    events: np.ndarray          # u32 [E]: bit31 = departure, bits 0..30 = request index
    event_off: np.ndarray       # u64 [n_streams+1]
    # weights: [n_streams] of (w_net, w_prefix, w_load)
    weights: np.ndarray         # f32 [n_streams, 3]

    @property
    def R(self) -> int:
        return int(self.length.shape[0])

    @property
    def n_streams(self) -> int:
        return int(self.req_off.shape[0] - 1)

    @property
    def capacity(self) -> int:
        return 1 << self.spec.log2_cap

    # ---- bulk arrays, host side ----
    def chains(self, r0: int = 0, r1: Optional[int] = None) -> np.ndarray:
        """Block-hash chains of requests [r0, r1), concatenated (offsets chain_off[r0..r1])."""
        r1 = self.R if r1 is None else r1
        out = []
        set_of = request_set(self)
        for r in range(r0, r1):
            n = int(self.chain_off[r + 1] - self.chain_off[r])
            out.append(chain_of(self, r, n, int(set_of[r])))
        return np.concatenate(out) if out else np.zeros(0, U64)

    def keys(self, g: int, d: int) -> np.ndarray:
        """Cached block hashes of decode d in table set g (insertion list)."""
        return cache_keys(self, g, d)

    def util(self, s0: int = 0, s1: Optional[int] = None, direction: str = "up") -> np.ndarray:
        s1 = self.n_snap if s1 is None else s1
        return utilisation(self, np.arange(s0, s1), direction)


def distinct_keys_per_group(w: Workload, group: int = 64) -> int:
    """Largest number of distinct cached hashes over (table set, group of `group`
    decodes): the union of the root prefixes plus every decode's filler keys."""
    best = 0
    for g in range(w.n_sets):
        for q0 in range(0, w.D, group):
            dd = w.depth[g, q0:q0 + group]
            best = max(best, int(dd.max(axis=0).sum() + (w.spec.n_keys - dd.sum(axis=1)).sum()))
    return best


def request_set(w: Workload) -> np.ndarray:
    out = np.zeros(w.R, np.int64)
    for g in range(w.n_sets):
        out[w.set_off[g]:w.set_off[g + 1]] = g
    return out


def constructed_hits(w: Workload, r0: int = 0, r1: Optional[int] = None) -> np.ndarray:
    """[r1 - r0, D] uint16: the leading run of cached blocks each (request, decode) has by
    construction.  A chain is the first `shared` blocks of its root followed by blocks no
    cache lists, and decode d of table set g lists the first depth[g, d, k] blocks of every
    root k, so the run is min(shared_r, depth[g, d, root_r]) (barring a 64-bit collision
    between independently drawn hashes)."""
    r1 = w.R if r1 is None else r1
    g = request_set(w)[r0:r1, None]
    dep = w.depth.astype(np.uint16)[g, np.arange(w.D)[None, :], w.root[r0:r1, None].astype(np.int64)]
    return np.minimum(w.shared[r0:r1, None].astype(np.uint16), dep)


def chain_of(w: Workload, r: int, n: int, g: int) -> np.ndarray:
    s = int(np.searchsorted(w.req_off, r, side="right") - 1)
    local = r - int(w.req_off[s])
    i = np.arange(n, dtype=np.int64)
    sh = int(w.shared[r])
    rootpart = nonzero_hash(draw(int(w.set_seed[g]), P_ROOTHASH, int(w.root[r]), i[:sh]))
    tail = nonzero_hash(draw(int(w.stream_seed[s]), P_TAIL, local, i[sh:]))
    return np.concatenate([rootpart, tail]).astype(U64)


def cache_keys(w: Workload, g: int, d: int) -> np.ndarray:
    spec = w.spec
    parts = []
    total = 0
    for k in range(spec.n_roots):
        dk = int(w.depth[g, d, k])
        parts.append(nonzero_hash(draw(int(w.set_seed[g]), P_ROOTHASH, k, np.arange(dk))))
        total += dk
    nf = spec.n_keys - total
    parts.append(nonzero_hash(draw(int(w.set_seed[g]), P_FILLER, d, np.arange(nf))))
    return np.concatenate(parts).astype(U64)


DOWN_SEED = 1 << 40  # downward utilisations (directed links) draw from seed + DOWN_SEED
TIER_SEED = 1 << 41  # per-tier congestion rows (the paper's four maps) from seed + TIER_SEED


def utilisation(w: Workload, snaps: np.ndarray, direction: str = "up") -> np.ndarray:
    """Utilisation rows of snapshots `snaps`.  direction "up" is the undirected row (and
    the upward one of directed links); "down" is an independent draw of the same
    distribution for the downward direction; "tiers" gives four per-tier congestion
    values per snapshot, uniform in [0, 0.9), for the paper's per-tier maps."""
    spec = w.spec
    snaps = np.asarray(snaps, dtype=np.int64)
    if direction == "tiers":  # draw(seed + TIER_SEED, P_UTIL, local index, tier), vectorised
        seeds = w.snap_seed[snaps].astype(np.int64) + TIER_SEED
        uniq, inv = np.unique(seeds, return_inverse=True)
        k = np.array([stream_key(int(x), P_UTIL) for x in uniq], dtype=U64)[inv.reshape(-1)]
        loc = w.snap_local[snaps].astype(U64)
        with np.errstate(over="ignore"):
            k2 = _mix(k + (loc + U64(1)) * U64(GOLDEN))
            vals = _mix(k2[:, None] + (np.arange(4, dtype=U64)[None, :] + U64(1)) * U64(GOLDEN))
        return uniform09_f32(vals).astype(np.float32).reshape(len(snaps), 4)
    e = np.arange(w.L, dtype=np.int64)
    out = np.empty((len(snaps), w.L), np.float32)
    shift = 0 if direction == "up" else DOWN_SEED
    for j, s in enumerate(snaps):
        seed = int(w.snap_seed[s]) + shift
        loc = int(w.snap_local[s])
        if spec.util_mode == "uniform09":
            out[j] = uniform09_f32(draw(seed, P_UTIL, loc, e))
        elif spec.util_mode == "beta25_hot":
            out[j] = beta25_hot_row(spec, seed, loc, w.L)
        else:
            raise ValueError(spec.util_mode)
    return out


def hot_links(spec: Spec, seed: int) -> np.ndarray:
    """5% of the used edges, fixed for the run: the ones with the smallest selection draws."""
    lu = used_links(spec)
    n_hot = int(round(0.05 * lu))
    key = draw(seed, P_HOTSEL, np.arange(lu), 0)
    return np.sort(np.argsort(key, kind="stable")[:n_hot])


def beta25_hot_row(spec: Spec, seed: int, s: int, L: int) -> np.ndarray:
    """Beta(2,5) = X/(X+Y), X ~ Gamma(2), Y ~ Gamma(5) as sums of -ln U; hot links U[0.85, 0.99]."""
    e = np.arange(L, dtype=np.int64)
    g = [-np.log1p(-unit(draw(seed, P_BETA, s, e * 8 + j))) for j in range(7)]
    x = g[0] + g[1]
    y = g[2] + g[3] + g[4] + g[5] + g[6]
    u = x / (x + y)
    hot = hot_links(spec, seed)
    u[hot] = 0.85 + 0.14 * unit(draw(seed, P_HOT, s, hot))
    u = u.astype(np.float32)
    return np.minimum(u, np.float32(np.nextafter(np.float32(1), np.float32(0))))


def stream_weights(spec: Spec, n_streams: int) -> np.ndarray:
    if spec.weights == "unit":
        return np.ones((n_streams, 3), np.float32)
    if spec.weights == "grid16":
        g = np.linspace(0.1, 2.0, 16).astype(np.float32)
        i = np.arange(n_streams)
        return np.stack([g[(i >> 8) & 15], g[(i >> 4) & 15], g[i & 15]], axis=1).astype(np.float32)
    raise ValueError(spec.weights)


def snapshot_of(arrival_us: np.ndarray) -> np.ndarray:
    """Telemetry refreshed every 100 ms and read 50 ms stale."""
    t = arrival_us.astype(np.int64)
    return np.where(t >= SNAP_STALE_US, (t - SNAP_STALE_US) // SNAP_PERIOD_US, 0)


def draw_rows(seed_per_row: np.ndarray, purpose: int, a: np.ndarray, b=0) -> np.ndarray:
    """draw(seed_per_row[i], purpose, a[i], b) for every row i (vectorised over seeds)."""
    seed_per_row = np.asarray(seed_per_row, dtype=np.int64)
    seeds, inv = np.unique(seed_per_row, return_inverse=True)
    k = np.array([stream_key(int(x), purpose) for x in seeds], dtype=U64)[inv.reshape(-1)]
    a = np.asarray(a, dtype=U64)
    b = np.asarray(b, dtype=U64)
    with np.errstate(over="ignore"):
        k2 = _mix(k + (a + U64(1)) * U64(GOLDEN))
        return _mix(k2 + (b + U64(1)) * U64(GOLDEN))


def make_workload(spec: Spec, n_streams: Optional[int] = None,
                  requests_per_stream: Optional[int] = None) -> Workload:
    """Materialise per-request arrays, events and depths; bulk arrays stay lazy."""
    role = roles(spec)
    P = int((role == 0).sum())
    D = int((role == 1).sum())
    L = n_links(spec)
    ns = spec.n_streams if n_streams is None else n_streams
    rps = spec.requests_per_stream if requests_per_stream is None else requests_per_stream
    seeds = np.arange(spec.seed0, spec.seed0 + ns, dtype=np.int64)
    R = ns * rps
    sidx = np.repeat(np.arange(ns, dtype=np.int64), rps)          # stream of each request
    sd = seeds[sidx]
    idx = np.tile(np.arange(rps, dtype=np.int64), ns)             # index within the stream
    req_off = np.arange(ns + 1, dtype=np.int64) * rps

    def lognorm(purpose, median, sigma):
        u1 = unit(draw_rows(sd, purpose, idx, 0))
        u2 = unit(draw_rows(sd, purpose, idx, 1))
        z = np.sqrt(-2.0 * np.log1p(-u1)) * np.cos(2.0 * np.pi * u2)
        return median * np.exp(sigma * z)

    if R:
        if spec.len_mode == "lognormal":
            ln = np.clip(np.rint(lognorm(P_LEN, spec.len_median, spec.len_sigma)),
                         spec.len_clip[0], spec.len_clip[1]).astype(np.int64)
        else:
            ln = np.full(R, spec.len_fixed, np.int64)
        out = np.clip(np.rint(lognorm(P_OUT, 256.0, 1.0)), 1, 4096).astype(np.int64)
        gap = np.rint(-np.log1p(-unit(draw_rows(sd, P_GAP, idx))) / spec.rate_per_s * 1e6).astype(np.int64)
        csum = np.cumsum(gap)
        base = np.concatenate([[0], csum[req_off[1:-1] - 1]]) if ns > 1 else np.zeros(1, np.int64)
        arrival = csum - base[sidx]
        prefill = below(draw_rows(sd, P_PREFILL, idx), P).astype(np.int64)
        root = below(draw_rows(sd, P_ROOT, idx), spec.n_roots).astype(np.int64)
        nb = ln // BLOCK_TOKENS
        rl = spec.root_len(root)
        if spec.share_mode == "frac":
            f = 0.9 * unit(draw_rows(sd, P_SHARE, idx))
            shared = np.minimum(np.floor(f * nb).astype(np.int64), rl)
        else:
            shared = np.minimum(rl, nb)
        depart = arrival + out * TBT_US
    else:
        ln = out = arrival = prefill = root = shared = depart = np.zeros(0, np.int64)
        nb = np.zeros(0, np.int64)

    length = ln.astype(np.uint32)
    chain_off = np.zeros(R + 1, np.uint64)
    chain_off[1:] = np.cumsum(nb.astype(np.uint64))

    # telemetry snapshots
    if spec.n_snapshots is not None:
        n_snap = spec.n_snapshots
        snap_seed = np.full(n_snap, spec.seed0, np.int64)
        snap_local = np.arange(n_snap, dtype=np.int64)
        snap = np.zeros(R, np.uint32)
    else:
        k = snapshot_of(arrival) if R else np.zeros(0, np.int64)
        if spec.telemetry == "per_stream":
            counts = (np.maximum.reduceat(k, req_off[:-1]) + 1) if R else np.ones(ns, np.int64)
            sbase = np.concatenate([[0], np.cumsum(counts)]).astype(np.int64)
            n_snap = int(sbase[-1])
            snap_seed = np.repeat(seeds, counts).astype(np.int64)
            snap_local = (np.arange(n_snap, dtype=np.int64) - np.repeat(sbase[:-1], counts))
            snap = (sbase[sidx] + k).astype(np.uint32)
        else:
            n_snap = int(k.max()) + 1 if R else 1
            snap_seed = np.full(n_snap, spec.seed0, np.int64)
            snap_local = np.arange(n_snap, dtype=np.int64)
            snap = k.astype(np.uint32)

    # table sets
    if spec.tables == "per_stream":
        n_sets = max(ns, 1)
        set_off = req_off.astype(np.uint32) if ns else np.zeros(2, np.uint32)
        set_seed = seeds.copy() if ns else np.array([spec.seed0], np.int64)
    else:
        n_sets = 1
        set_off = np.array([0, R], np.uint32)
        set_seed = np.array([spec.seed0], np.int64)
    kk = np.arange(spec.n_roots, dtype=np.int64)
    rl = spec.root_len(kk)
    gg = np.repeat(np.arange(n_sets), D * spec.n_roots)
    dd = np.tile(np.repeat(np.arange(D), spec.n_roots), n_sets)
    kx = np.tile(kk, n_sets * D)
    raw = below(draw_rows(set_seed[gg], P_DEPTH, dd, kx), (rl[kx] + 1).astype(np.uint64))
    depth = raw.astype(np.int64).reshape(n_sets, D, spec.n_roots)
    if spec.depth_mode == "scaled":
        tot = depth.sum(axis=2, keepdims=True)
        depth = np.where(tot > spec.n_keys, (depth * spec.n_keys) // np.maximum(tot, 1), depth)
    assert (depth.sum(axis=2) <= spec.n_keys).all()

    # events: per stream, sorted by (time, departure before arrival, request index)
    if R:
        rr = np.concatenate([np.arange(R), np.arange(R)])
        t = np.concatenate([depart, arrival])
        typ = np.concatenate([np.zeros(R, np.int64), np.ones(R, np.int64)])
        order = np.lexsort((rr, typ, t, sidx[rr]))
        events = (rr[order].astype(np.uint64) |
                  ((1 - typ[order]).astype(np.uint64) << U64(31))).astype(np.uint32)
    else:
        events = np.zeros(0, np.uint32)
    event_off = (np.arange(ns + 1, dtype=np.uint64) * np.uint64(2 * rps))

    return Workload(spec=spec, role=role, P=P, D=D, L=L, req_off=req_off, stream_seed=seeds,
                    length=length, prefill=prefill.astype(np.uint32), arrival_us=arrival,
                    depart_us=depart, snap=snap, root=root.astype(np.uint32),
                    shared=shared.astype(np.uint32), chain_off=chain_off, n_sets=n_sets,
                    set_off=set_off, set_seed=set_seed, depth=depth, n_snap=n_snap,
                    snap_seed=snap_seed, snap_local=snap_local, events=events,
                    event_off=event_off, weights=stream_weights(spec, ns))


def tiny_spec(**kw) -> Spec:
    """Small four-tier tree with fanouts (2,2,2,2) so that every tier occurs."""
    base = dict(name="tiny", fanout=(2, 2, 2, 2), role_rule="alternate", n_streams=2,
                requests_per_stream=40, rate_per_s=50.0, len_median=2048.0,
                len_clip=(16, 16384), n_roots=4, root_blocks=(1024,), n_keys=3000,
                log2_cap=12, tables="per_stream", telemetry="per_stream",
                cap_tokens=40_000)
    base.update(kw)
    return Spec(**base)
