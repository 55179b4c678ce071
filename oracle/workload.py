"""Run the CPU oracle on generated workloads, one stream at a time.

TEST INFRASTRUCTURE ONLY (tests, smoke check, benchmark CPU baseline).

A stream is made self-contained: its requests are renumbered from 0, its events
re-encoded, its telemetry rows gathered.  ``stream_inputs`` does that gathering (the
generator's output, no arithmetic of the method); the oracle then computes the prefix
hits (by set membership over the generator's key lists), the greedy and, for the
tests, the level bottlenecks, all in double precision.  The benchmark times the
oracle alone by preparing the inputs first (``stream_inputs``) and timing
``solve_stream``.
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import numpy as np

from . import (level_bottleneck_directed, prefix_match, schedule_stream, schedule_stream_evolving,
               schedule_stream_inflight, schedule_stream_load, up_bottleneck)


@dataclasses.dataclass
class OracleStream:
    r0: int
    r1: int
    M: np.ndarray          # [R_s, D] uint16
    dec: np.ndarray        # [R_s] int32
    best: np.ndarray       # [R_s] float64
    second: np.ndarray     # [R_s] float64
    load: np.ndarray       # [D] int64
    near_ties: int
    mismatches: int
    rejects: int
    snaps: np.ndarray      # global snapshot indices used by the stream's arrivals
    UB: np.ndarray         # [len(snaps), N, 4] oracle level bottlenecks of those snapshots


@dataclasses.dataclass
class StreamInputs:
    """One stream's inputs, gathered from the generator (requests renumbered from 0)."""
    s: int
    r0: int
    r1: int
    ev_local: np.ndarray           # u32 events with local request indices
    snaps: np.ndarray              # global snapshot indices used by the stream's arrivals
    snap_local: np.ndarray         # u32 [R_s] index into util
    util: np.ndarray               # f32 [len(snaps), L] (or [len(snaps), 4] per tier)
    util_down: Optional[np.ndarray]
    keys: Optional[np.ndarray]     # the stream's caches: key lists of its table set
    key_off: Optional[np.ndarray]
    chains: Optional[np.ndarray]   # the stream's chains, offsets from 0
    chain_off: Optional[np.ndarray]
    M: Optional[np.ndarray]        # given prefix hits (then no keys or chains)


def stream_problem(w, s: int):
    r0, r1 = int(w.req_off[s]), int(w.req_off[s + 1])
    e0, e1 = int(w.event_off[s]), int(w.event_off[s + 1])
    ev = w.events[e0:e1].astype(np.uint64)
    r_local = (ev & np.uint64(0x7FFFFFFF)) - np.uint64(r0)
    ev_local = (r_local | (ev & np.uint64(1 << 31))).astype(np.uint32)
    snaps, snap_local = np.unique(w.snap[r0:r1].astype(np.int64), return_inverse=True)
    return r0, r1, ev_local, snaps, snap_local.astype(np.uint32)


def stream_cache_keys(w, g: int):
    keys = [w.keys(g, d) for d in range(w.D)]
    off = np.concatenate([[0], np.cumsum([len(k) for k in keys])]).astype(np.uint64)
    return np.concatenate(keys), off


def _rows(w, snaps, direction):
    if w.n_snap * w.L < (1 << 24):
        return w.util(direction=direction)[snaps]
    return np.stack([w.util(int(k), int(k) + 1, direction)[0] for k in snaps])


def stream_inputs(w, s: int, M: Optional[np.ndarray] = None, directed: bool = False,
                  tiers: bool = False) -> StreamInputs:
    """Gather stream s's inputs from the generator: events, telemetry rows, and either the
    given prefix hits M or the key lists and chains the oracle matches itself."""
    from synth import request_set, utilisation
    r0, r1, ev_local, snaps, snap_local = stream_problem(w, s)
    util = utilisation(w, snaps, "tiers") if tiers else _rows(w, snaps, "up")
    util_down = _rows(w, snaps, "down") if directed else None
    keys = key_off = chains = chain_off = None
    if M is None:
        g = int(request_set(w)[r0]) if r1 > r0 else 0
        keys, key_off = stream_cache_keys(w, g)
        chains = w.chains(r0, r1)
        chain_off = (w.chain_off[r0:r1 + 1] - w.chain_off[r0]).astype(np.uint64)
    return StreamInputs(s, r0, r1, ev_local, snaps, snap_local, util, util_down, keys, key_off,
                        chains, chain_off, M)


def stream_hits(w, x: StreamInputs) -> np.ndarray:
    """The oracle's prefix hits of the stream (or the given ones)."""
    if x.M is not None:
        return x.M
    return prefix_match(x.keys, x.key_off, w.D, x.chains, x.chain_off,
                        np.array([0, x.r1 - x.r0], np.uint32))


def solve_stream(w, x: StreamInputs, theta: float, cap: int, bytes_per_token: int,
                 inflight_cap: int = 0, load_model=None, tiers: bool = False):
    """The oracle's work for one prepared stream: its prefix match and its greedy (with
    self-contention when inflight_cap > 0, with the compute-load model when load_model =
    (t_a, t_b, beta_max, m_min, m0) is given).  Returns (M, greedy result)."""
    M = stream_hits(w, x)
    wn, wp, wl = (float(v) for v in w.weights[x.s])
    spec = w.spec
    r0, r1 = x.r0, x.r1
    if load_model is not None:
        a, b, bmax, m_min, m0 = load_model
        res = schedule_stream_load(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, x.util,
                                   w.length[r0:r1], w.prefill[r0:r1], x.snap_local, M, x.ev_local,
                                   wn, wp, wl, bytes_per_token, a, b, bmax, m_min, m0)
    elif inflight_cap > 0:
        res = schedule_stream_inflight(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, x.util,
                                       w.length[r0:r1], w.prefill[r0:r1], x.snap_local,
                                       w.arrival_us[r0:r1], M, x.ev_local, wn, wp, wl, theta, cap,
                                       bytes_per_token, inflight_cap)
    else:
        res = schedule_stream(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, x.util,
                              w.length[r0:r1], w.prefill[r0:r1], x.snap_local, M, x.ev_local,
                              wn, wp, wl, theta, cap, bytes_per_token, util_down=x.util_down,
                              tier_mode=tiers)
    return M, res


def run_stream(w, s: int, theta: float, cap: int, bytes_per_token: int,
               hint: Optional[np.ndarray] = None, rel_tol: float = 1e-5,
               M: Optional[np.ndarray] = None, directed: bool = False,
               tiers: bool = False) -> OracleStream:
    """Oracle for stream s of workload w (per-stream table sets and telemetry, or shared).

    hint: decisions of another implementation for this stream's requests (local order).
    directed: links carry separate upward and downward utilisations (the generator's
    "up" and "down" rows); UB is then the directed level bottleneck.
    tiers: the paper's per-tier maps (the generator's "tiers" rows, four congestion
    values per snapshot); UB[s][i][k] is then B_k (1 - c[s][k]) for every instance.
    """
    x = stream_inputs(w, s, M=M, directed=directed, tiers=tiers)
    M = stream_hits(w, x)
    r0, r1 = x.r0, x.r1
    wn, wp, wl = (float(v) for v in w.weights[s])
    spec = w.spec
    res = schedule_stream(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, x.util,
                          w.length[r0:r1], w.prefill[r0:r1], x.snap_local, M, x.ev_local,
                          wn, wp, wl, theta, cap, bytes_per_token, hint=hint, rel_tol=rel_tol,
                          util_down=x.util_down, tier_mode=tiers)
    if tiers:
        per_tier = np.asarray(spec.tier_bw, np.float64) * (1.0 - x.util.astype(np.float64))
        UB = np.repeat(per_tier[:, None, :], len(w.role), axis=1)
    elif directed:
        UB = level_bottleneck_directed(spec.fanout, w.role, spec.tier_bw, x.util, x.util_down)
    else:
        UB = up_bottleneck(spec.fanout, spec.tier_bw, x.util)
    return OracleStream(r0, r1, M, res.dec, res.best, res.second, res.load, res.near_ties,
                        res.mismatches, res.rejects, x.snaps, UB)


def run_stream_inflight(w, s: int, theta: float, cap: int, bytes_per_token: int,
                        inflight_cap: int, hint: Optional[np.ndarray] = None,
                        xfer_hint: Optional[np.ndarray] = None, rel_tol: float = 1e-5,
                        M: Optional[np.ndarray] = None) -> OracleStream:
    """Oracle for stream s with self-contention (Eq. 4's n_inflight, Algorithm 1 lines 5
    and 14).  hint / xfer_hint: another implementation's decisions and transfer times
    for the stream's requests (local order).  The result carries xfer_us."""
    x = stream_inputs(w, s, M=M)
    M = stream_hits(w, x)
    r0, r1 = x.r0, x.r1
    wn, wp, wl = (float(v) for v in w.weights[s])
    spec = w.spec
    res = schedule_stream_inflight(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, x.util,
                                   w.length[r0:r1], w.prefill[r0:r1], x.snap_local,
                                   w.arrival_us[r0:r1], M, x.ev_local, wn, wp, wl, theta, cap,
                                   bytes_per_token, inflight_cap, hint=hint, xfer_hint=xfer_hint,
                                   rel_tol=rel_tol)
    UB = up_bottleneck(spec.fanout, spec.tier_bw, x.util)
    out = OracleStream(r0, r1, M, res.dec, res.best, res.second, res.load, res.near_ties,
                       res.mismatches, res.rejects, x.snaps, UB)
    out.xfer_us, out.xfer_adopted, out.xfer_mismatches = res.xfer_us, res.xfer_adopted, res.xfer_mismatches
    return out


def run_stream_load(w, s: int, t_a: float, t_b: float, beta_max: int, m_min: int, m0: int,
                    bytes_per_token: int, hint: Optional[np.ndarray] = None,
                    rel_tol: float = 1e-5, M: Optional[np.ndarray] = None):
    """Oracle for stream s with the paper's compute-load model (Sec. III-C, IV-B); hint: another
    implementation's decisions for the stream's requests (local order).  Returns the
    oracle's LoadResult with its prefix hits attached (.M)."""
    x = stream_inputs(w, s, M=M)
    M = stream_hits(w, x)
    r0, r1 = x.r0, x.r1
    wn, wp, wl = (float(v) for v in w.weights[s])
    spec = w.spec
    res = schedule_stream_load(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, x.util,
                               w.length[r0:r1], w.prefill[r0:r1], x.snap_local, M, x.ev_local, wn,
                               wp, wl, bytes_per_token, t_a, t_b, beta_max, m_min, m0, hint=hint,
                               rel_tol=rel_tol)
    res.M = M
    return res


def run_stream_evolving(w, s: int, theta: float, cap: int, bytes_per_token: int, cap_blocks: int,
                        hint: Optional[np.ndarray] = None, rel_tol: float = 1e-5):
    """Oracle for stream s with evolving LRU caches of cap_blocks blocks (Sec. VI-B): the
    stream's decodes start from its table set's key lists, most recently used first.
    hint: another implementation's decisions (local order).  Returns the oracle's
    EvolvingResult (hits per arrival .M, final caches .caches)."""
    x = stream_inputs(w, s)
    r0, r1 = x.r0, x.r1
    wn, wp, wl = (float(v) for v in w.weights[s])
    spec = w.spec
    return schedule_stream_evolving(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, x.util,
                                    w.length[r0:r1], w.prefill[r0:r1], x.snap_local, x.keys,
                                    x.key_off, x.chains, x.chain_off, x.ev_local, wn, wp, wl,
                                    theta, cap, bytes_per_token, hint=hint, rel_tol=rel_tol,
                                    cap_blocks=cap_blocks)
