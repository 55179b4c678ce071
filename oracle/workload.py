"""Run the CPU oracle on generated workloads, one stream at a time.

TEST INFRASTRUCTURE ONLY (tests, smoke check, benchmark CPU baseline).

A stream is made self-contained: its requests are renumbered from 0, its events
re-encoded, its telemetry rows gathered; the oracle then computes the level
bottlenecks, the prefix hits (by set membership over the generator's key
lists) and the greedy, all in double precision.
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import numpy as np

from . import (level_bottleneck_directed, prefix_match, schedule_stream, schedule_stream_inflight,
               schedule_stream_load, up_bottleneck)


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
    from synth import request_set, utilisation
    r0, r1, ev_local, snaps, snap_local = stream_problem(w, s)
    util = utilisation(w, snaps, "tiers") if tiers else _rows(w, snaps, "up")
    util_down = _rows(w, snaps, "down") if directed else None
    if M is None:
        g = int(request_set(w)[r0]) if r1 > r0 else 0
        keys, key_off = stream_cache_keys(w, g)
        chains = w.chains(r0, r1)
        chain_off = (w.chain_off[r0:r1 + 1] - w.chain_off[r0]).astype(np.uint64)
        M = prefix_match(keys, key_off, w.D, chains, chain_off,
                         np.array([0, r1 - r0], np.uint32))
    wn, wp, wl = (float(x) for x in w.weights[s])
    spec = w.spec
    res = schedule_stream(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, util,
                          w.length[r0:r1], w.prefill[r0:r1], snap_local, M, ev_local,
                          wn, wp, wl, theta, cap, bytes_per_token, hint=hint, rel_tol=rel_tol,
                          util_down=util_down, tier_mode=tiers)
    if tiers:
        per_tier = np.asarray(spec.tier_bw, np.float64) * (1.0 - util.astype(np.float64))
        UB = np.repeat(per_tier[:, None, :], len(w.role), axis=1)
    elif directed:
        UB = level_bottleneck_directed(spec.fanout, w.role, spec.tier_bw, util, util_down)
    else:
        UB = up_bottleneck(spec.fanout, spec.tier_bw, util)
    return OracleStream(r0, r1, M, res.dec, res.best, res.second, res.load, res.near_ties,
                        res.mismatches, res.rejects, snaps, UB)


def run_stream_inflight(w, s: int, theta: float, cap: int, bytes_per_token: int,
                        inflight_cap: int, hint: Optional[np.ndarray] = None,
                        xfer_hint: Optional[np.ndarray] = None, rel_tol: float = 1e-5,
                        M: Optional[np.ndarray] = None) -> OracleStream:
    """Oracle for stream s with self-contention (Eq. 4's n_inflight, Algorithm 1 lines 5
    and 14).  hint / xfer_hint: another implementation's decisions and transfer times
    for the stream's requests (local order).  The result carries xfer_us."""
    from synth import request_set, utilisation
    r0, r1, ev_local, snaps, snap_local = stream_problem(w, s)
    util = _rows(w, snaps, "up")
    if M is None:
        g = int(request_set(w)[r0]) if r1 > r0 else 0
        keys, key_off = stream_cache_keys(w, g)
        chains = w.chains(r0, r1)
        chain_off = (w.chain_off[r0:r1 + 1] - w.chain_off[r0]).astype(np.uint64)
        M = prefix_match(keys, key_off, w.D, chains, chain_off,
                         np.array([0, r1 - r0], np.uint32))
    wn, wp, wl = (float(x) for x in w.weights[s])
    spec = w.spec
    res = schedule_stream_inflight(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, util,
                                   w.length[r0:r1], w.prefill[r0:r1], snap_local,
                                   w.arrival_us[r0:r1], M, ev_local, wn, wp, wl, theta, cap,
                                   bytes_per_token, inflight_cap, hint=hint, xfer_hint=xfer_hint,
                                   rel_tol=rel_tol)
    UB = up_bottleneck(spec.fanout, spec.tier_bw, util)
    out = OracleStream(r0, r1, M, res.dec, res.best, res.second, res.load, res.near_ties,
                       res.mismatches, res.rejects, snaps, UB)
    out.xfer_us, out.xfer_adopted, out.xfer_mismatches = res.xfer_us, res.xfer_adopted, res.xfer_mismatches
    return out


def run_stream_load(w, s: int, t_a: float, t_b: float, beta_max: int, m_min: int, m0: int,
                    bytes_per_token: int, hint: Optional[np.ndarray] = None,
                    rel_tol: float = 1e-5, M: Optional[np.ndarray] = None):
    """Oracle for stream s with the paper's compute-load model (Sec. III-C, IV-B); hint: another
    implementation's decisions for the stream's requests (local order).  Returns the
    oracle's LoadResult with its prefix hits attached (.M)."""
    from synth import request_set
    r0, r1, ev_local, snaps, snap_local = stream_problem(w, s)
    util = _rows(w, snaps, "up")
    if M is None:
        g = int(request_set(w)[r0]) if r1 > r0 else 0
        keys, key_off = stream_cache_keys(w, g)
        chains = w.chains(r0, r1)
        chain_off = (w.chain_off[r0:r1 + 1] - w.chain_off[r0]).astype(np.uint64)
        M = prefix_match(keys, key_off, w.D, chains, chain_off,
                         np.array([0, r1 - r0], np.uint32))
    wn, wp, wl = (float(x) for x in w.weights[s])
    spec = w.spec
    res = schedule_stream_load(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, util,
                               w.length[r0:r1], w.prefill[r0:r1], snap_local, M, ev_local, wn, wp,
                               wl, bytes_per_token, t_a, t_b, beta_max, m_min, m0, hint=hint,
                               rel_tol=rel_tol)
    res.M = M
    return res
