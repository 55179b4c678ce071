"""Python loader for the NetKV CPU oracle (``netkv_oracle.cpp``).

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()`` and
the benchmark's CPU-baseline leg.  The product path never imports this package.

The oracle is plain C++ in double precision compiled with g++ (OpenMP across
independent units only).  ``build()`` compiles it; the functions below marshal
numpy arrays to it and return numpy results.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
from typing import Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "netkv_oracle.cpp")
_LIB = os.path.join(_HERE, "libnetkv_oracle.so")
_lib = None


def build(force: bool = False) -> str:
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["g++", "-O2", "-std=c++17", "-fopenmp", "-shared", "-fPIC",
                               _SRC, "-o", tmp])
        os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    if _lib is None:
        build()
        _lib = C.CDLL(_LIB)
        _declare(_lib)
    return _lib


P = C.c_void_p
U32, U64, I64, F64, INT = C.c_uint32, C.c_uint64, C.c_int64, C.c_double, C.c_int


def _declare(l):
    l.oracle_set_threads.restype = None
    l.oracle_set_threads.argtypes = [INT]
    l.oracle_kv_bytes_per_token.restype = F64
    l.oracle_kv_bytes_per_token.argtypes = [U32, U32, U32, U32]
    l.oracle_beff_tier.restype = F64
    l.oracle_beff_tier.argtypes = [F64, F64, F64]
    l.oracle_transfer_time.restype = F64
    l.oracle_transfer_time.argtypes = [F64, F64, F64]
    l.oracle_s_eff.restype = F64
    l.oracle_s_eff.argtypes = [F64, F64, F64]
    l.oracle_tier.restype = INT
    l.oracle_tier.argtypes = [P, U64, U64]
    l.oracle_path_links.restype = INT
    l.oracle_path_links.argtypes = [P, U64, U64, P, P]
    l.oracle_used_links.restype = U64
    l.oracle_used_links.argtypes = [P]
    l.oracle_cost_matrix.restype = None
    l.oracle_cost_matrix.argtypes = [P, P, P, P, P, U64, U64, F64, P]
    l.oracle_cost_entries.restype = None
    l.oracle_cost_entries.argtypes = [P, P, P, P, P, U64, P, P, P, U64, F64, P]
    l.oracle_up_bottleneck.restype = None
    l.oracle_up_bottleneck.argtypes = [P, P, P, U64, U64, P]
    l.oracle_prefix_match.restype = None
    l.oracle_prefix_match.argtypes = [P, P, U32, P, P, U32, P, U32, P]
    l.oracle_prefix_match_one.restype = None
    l.oracle_prefix_match_one.argtypes = [P, U64, P, P, U64, P]
    l.oracle_schedule_stream.restype = None
    l.oracle_schedule_stream.argtypes = [P, P, P, P, P, P, INT, U64, P, P, P, P, P, U64, F64, F64,
                                         F64, F64, I64, U64, P, P, F64, P, P, P, P, P]
    l.oracle_schedule_stream_load.restype = None
    l.oracle_schedule_stream_load.argtypes = [P, P, P, P, P, U64, P, P, P, P, P, U64, F64, F64,
                                              F64, U64, F64, F64, I64, I64, I64, P, P, P, F64,
                                              P, P, P, P, P, P]
    l.oracle_schedule_stream_evolving.restype = None
    l.oracle_schedule_stream_evolving.argtypes = [P, P, P, P, P, U64, P, P, P, P, P, U64, P, P, P,
                                                  U64, F64, F64, F64, F64, I64, U64, P, F64, P, P,
                                                  P, P, P, P, P, U64, P]
    l.oracle_cost_matrix_tiers.restype = None
    l.oracle_cost_matrix_tiers.argtypes = [P, P, P, P, P, U64, F64, P]
    l.oracle_cost_matrix_directed.restype = None
    l.oracle_cost_matrix_directed.argtypes = [P, P, P, P, P, P, U64, U64, F64, P]
    l.oracle_level_bottleneck_directed.restype = None
    l.oracle_level_bottleneck_directed.argtypes = [P, P, P, P, P, U64, U64, P]
    l.oracle_schedule_stream_inflight.restype = None
    l.oracle_schedule_stream_inflight.argtypes = [P, P, P, P, P, U64, P, P, P, P, P, P, U64,
                                                  F64, F64, F64, F64, I64, U64, U32, P, P, P,
                                                  F64, P, P, P, P, P, P]


def _p(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _c(a, dt):
    return np.ascontiguousarray(np.asarray(a, dtype=dt))


def set_threads(n: int) -> None:
    """OpenMP threads of the calling thread's later oracle calls (timing only)."""
    lib().oracle_set_threads(int(n))


# ------------------------------------------------------------------ closed forms
def kv_bytes_per_token(n_layers=80, n_kv_heads=8, d_head=128, b_elem=2) -> float:
    return lib().oracle_kv_bytes_per_token(n_layers, n_kv_heads, d_head, b_elem)


def beff_tier(B, c, n_inflight=0.0) -> float:
    return lib().oracle_beff_tier(B, c, n_inflight)


def transfer_time(s, B_eff, L=0.0) -> float:
    return lib().oracle_transfer_time(s, B_eff, L)


def s_eff(s_r, lam, l_r) -> float:
    return lib().oracle_s_eff(s_r, lam, l_r)


# ------------------------------------------------------------------ topology
def tier(fanout: Sequence[int], i: int, j: int) -> int:
    f = _c(fanout, np.uint32)
    return lib().oracle_tier(_p(f), i, j)


def path_links(fanout: Sequence[int], i: int, j: int):
    f = _c(fanout, np.uint32)
    links = np.zeros(8, np.uint64)
    levels = np.zeros(8, np.int32)
    n = lib().oracle_path_links(_p(f), i, j, _p(links), _p(levels))
    return links[:n], levels[:n]


def used_links(fanout) -> int:
    f = _c(fanout, np.uint32)
    return int(lib().oracle_used_links(_p(f)))


# ------------------------------------------------------------------ oracle matrix
def cost_matrix(fanout, role, bw, lat, util, kv_bytes) -> np.ndarray:
    f, ro = _c(fanout, np.uint32), _c(role, np.uint8)
    b, la = _c(bw, np.float64), _c(lat, np.float64)
    u = _c(util, np.float32)
    S, L = u.shape
    P = int((ro == 0).sum()); D = int((ro == 1).sum())
    out = np.zeros((S, P, D), np.float64)
    lib().oracle_cost_matrix(_p(f), _p(ro), _p(b), _p(la), _p(u), L, S, float(kv_bytes), _p(out))
    return out


def cost_entries(fanout, role, bw, lat, util, s, p, d, kv_bytes) -> np.ndarray:
    f, ro = _c(fanout, np.uint32), _c(role, np.uint8)
    b, la = _c(bw, np.float64), _c(lat, np.float64)
    u = _c(util, np.float32)
    s, p, d = _c(s, np.uint64), _c(p, np.uint64), _c(d, np.uint64)
    out = np.zeros(len(s), np.float64)
    lib().oracle_cost_entries(_p(f), _p(ro), _p(b), _p(la), _p(u), u.shape[1], _p(s), _p(p),
                              _p(d), len(s), float(kv_bytes), _p(out))
    return out


def cost_matrix_directed(fanout, role, bw, lat, util_up, util_down, kv_bytes) -> np.ndarray:
    """C[s][p][d] with directed links: the prefill's links at their upward utilisation,
    the decode's at their downward one."""
    f, ro = _c(fanout, np.uint32), _c(role, np.uint8)
    b, la = _c(bw, np.float64), _c(lat, np.float64)
    uu, ud = _c(util_up, np.float32), _c(util_down, np.float32)
    assert uu.shape == ud.shape
    S, L = uu.shape
    P = int((ro == 0).sum()); D = int((ro == 1).sum())
    out = np.zeros((S, P, D), np.float64)
    lib().oracle_cost_matrix_directed(_p(f), _p(ro), _p(b), _p(la), _p(uu), _p(ud), L, S,
                                      float(kv_bytes), _p(out))
    return out


def cost_matrix_tiers(fanout, role, bw, lat, c, kv_bytes) -> np.ndarray:
    """C[s][p][d] of the paper-literal per-tier oracle: kv / (B_tau (1 - c[s][tau])) + L_tau."""
    f, ro = _c(fanout, np.uint32), _c(role, np.uint8)
    b, la = _c(bw, np.float64), _c(lat, np.float64)
    cc = _c(c, np.float32)
    S = cc.shape[0]
    assert cc.shape == (S, 4)
    P = int((ro == 0).sum()); D = int((ro == 1).sum())
    out = np.zeros((S, P, D), np.float64)
    lib().oracle_cost_matrix_tiers(_p(f), _p(ro), _p(b), _p(la), _p(cc), S, float(kv_bytes), _p(out))
    return out


def level_bottleneck_directed(fanout, role, bw, util_up, util_down) -> np.ndarray:
    """UB[s][i][k] with directed links: prefill instances at upward, decode instances at
    downward utilisation."""
    f, ro, b = _c(fanout, np.uint32), _c(role, np.uint8), _c(bw, np.float64)
    uu, ud = _c(util_up, np.float32), _c(util_down, np.float32)
    S, L = uu.shape
    out = np.zeros((S, len(ro), 4), np.float64)
    lib().oracle_level_bottleneck_directed(_p(f), _p(ro), _p(b), _p(uu), _p(ud), L, S, _p(out))
    return out


def up_bottleneck(fanout, bw, util) -> np.ndarray:
    f, b, u = _c(fanout, np.uint32), _c(bw, np.float64), _c(util, np.float32)
    S, L = u.shape
    n = int(np.prod(np.asarray(fanout, dtype=np.int64)))
    out = np.zeros((S, n, 4), np.float64)
    lib().oracle_up_bottleneck(_p(f), _p(b), _p(u), L, S, _p(out))
    return out


# ------------------------------------------------------------------ prefix match
def prefix_match(keys, key_off, D, chains, chain_off, set_off) -> np.ndarray:
    k, ko = _c(keys, np.uint64), _c(key_off, np.uint64)
    ch, co = _c(chains, np.uint64), _c(chain_off, np.uint64)
    so = _c(set_off, np.uint32)
    R = len(co) - 1
    out = np.zeros((R, D), np.uint16)
    lib().oracle_prefix_match(_p(k), _p(ko), D, _p(ch), _p(co), R, _p(so), len(so) - 1, _p(out))
    return out


def prefix_match_one(keys, chains, chain_off) -> np.ndarray:
    k = _c(keys, np.uint64)
    ch, co = _c(chains, np.uint64), _c(chain_off, np.uint64)
    out = np.zeros(len(co) - 1, np.uint16)
    lib().oracle_prefix_match_one(_p(k), len(k), _p(ch), _p(co), len(co) - 1, _p(out))
    return out


# ------------------------------------------------------------------ greedy
class StreamResult:
    def __init__(self, dec, best, second, load, near_ties, mismatches, rejects, xfer_us=None,
                 xfer_adopted=0, xfer_mismatches=0):
        self.dec, self.best, self.second, self.load = dec, best, second, load
        self.near_ties, self.mismatches, self.rejects = near_ties, mismatches, rejects
        self.xfer_us, self.xfer_adopted, self.xfer_mismatches = xfer_us, xfer_adopted, xfer_mismatches


def schedule_stream(fanout, role, bw, lat, util, length, prefill, snap, M, events,
                    w_net, w_prefix, w_load, theta, cap, bytes_per_token,
                    load_init=None, hint=None, rel_tol=1e-5, dec_inout=None,
                    util_down=None, tier_mode=False) -> StreamResult:
    """Run one stream's events.  Arrays are indexed by global request index r.

    ``dec_inout`` (int32 [R]) carries decisions across streams that share request
    arrays; entries for this stream's requests are written.
    """
    f, ro = _c(fanout, np.uint32), _c(role, np.uint8)
    b, la = _c(bw, np.float64), _c(lat, np.float64)
    u = _c(util, np.float32)
    ln, pf, sn = _c(length, np.uint32), _c(prefill, np.uint32), _c(snap, np.uint32)
    m = _c(M, np.uint16)
    ev = _c(events, np.uint32)
    R = len(ln)
    D = int((ro == 1).sum())
    dec = np.full(R, -1, np.int32) if dec_inout is None else dec_inout
    best = np.full(R, np.inf); second = np.full(R, np.inf)
    load = np.zeros(D, np.int64)
    counts = np.zeros(3, np.int64)
    li = None if load_init is None else _c(load_init, np.int64)
    h = None if hint is None else _c(hint, np.int32)
    ud = None if util_down is None else _c(util_down, np.float32)
    assert ud is None or ud.shape == u.shape
    assert not tier_mode or u.shape[1] == 4
    lib().oracle_schedule_stream(_p(f), _p(ro), _p(b), _p(la), _p(u), _p(ud), int(bool(tier_mode)),
                                 u.shape[1], _p(ln), _p(pf),
                                 _p(sn), _p(m), _p(ev), len(ev), float(w_net), float(w_prefix),
                                 float(w_load), float(theta), int(cap), int(bytes_per_token),
                                 _p(li), _p(h), float(rel_tol), _p(dec), _p(best), _p(second),
                                 _p(load), _p(counts))
    return StreamResult(dec, best, second, load, int(counts[0]), int(counts[1]), int(counts[2]))


def schedule_stream_inflight(fanout, role, bw, lat, util, length, prefill, snap, arrival_us, M,
                             events, w_net, w_prefix, w_load, theta, cap, bytes_per_token,
                             inflight_cap, load_init=None, hint=None, xfer_hint=None,
                             rel_tol=1e-5) -> StreamResult:
    """Algorithm 1 with self-contention (Eq. 4's n_inflight, Algorithm 1 lines 5 and 14,
    Sec. V-C): arrays are indexed by request; arrival_us are the arrival times in
    microseconds; inflight_cap = 0 turns self-contention off.  xfer_hint: another
    implementation's transfer times (whole microseconds) to adopt where they differ by at
    most one.  Returns a StreamResult with xfer_us set."""
    f, ro = _c(fanout, np.uint32), _c(role, np.uint8)
    b, la = _c(bw, np.float64), _c(lat, np.float64)
    u = _c(util, np.float32)
    ln, pf, sn = _c(length, np.uint32), _c(prefill, np.uint32), _c(snap, np.uint32)
    ta = _c(arrival_us, np.int64)
    m = _c(M, np.uint16)
    ev = _c(events, np.uint32)
    R = len(ln)
    D = int((ro == 1).sum())
    dec = np.full(R, -1, np.int32)
    best = np.full(R, np.inf); second = np.full(R, np.inf)
    xfer = np.full(R, -1, np.int32)
    load = np.zeros(D, np.int64)
    counts = np.zeros(5, np.int64)
    li = None if load_init is None else _c(load_init, np.int64)
    h = None if hint is None else _c(hint, np.int32)
    xh = None if xfer_hint is None else _c(xfer_hint, np.int32)
    lib().oracle_schedule_stream_inflight(
        _p(f), _p(ro), _p(b), _p(la), _p(u), u.shape[1], _p(ln), _p(pf), _p(sn), _p(ta), _p(m),
        _p(ev), len(ev), float(w_net), float(w_prefix), float(w_load), float(theta), int(cap),
        int(bytes_per_token), int(inflight_cap), _p(li), _p(h), _p(xh), float(rel_tol), _p(dec),
        _p(best), _p(second), _p(xfer), _p(load), _p(counts))
    return StreamResult(dec, best, second, load, int(counts[0]), int(counts[1]), int(counts[2]),
                        xfer, int(counts[3]), int(counts[4]))


class LoadResult(StreamResult):
    def __init__(self, dec, best, second, n, m, near_ties, mismatches, rejects):
        super().__init__(dec, best, second, None, near_ties, mismatches, rejects)
        self.n, self.m = n, m


def schedule_stream_load(fanout, role, bw, lat, util, length, prefill, snap, M, events, w_net,
                         w_prefix, w_load, bytes_per_token, t_a, t_b, beta_max, m_min, m0,
                         m_init=None, n_init=None, hint=None, rel_tol=1e-5) -> LoadResult:
    """Algorithm 1 with the paper's compute-load model (Sec. III-C, IV-B): load term
    T_queue + T_decode from each decode's request count with t_iter(beta) = t_a + t_b beta,
    feasibility m_d >= s_eff + m_min.  Returns decisions, scores and the final request
    counts and free memory per decode."""
    f, ro = _c(fanout, np.uint32), _c(role, np.uint8)
    b, la = _c(bw, np.float64), _c(lat, np.float64)
    u = _c(util, np.float32)
    ln, pf, sn = _c(length, np.uint32), _c(prefill, np.uint32), _c(snap, np.uint32)
    mm = _c(M, np.uint16)
    ev = _c(events, np.uint32)
    R = len(ln)
    D = int((ro == 1).sum())
    dec = np.full(R, -1, np.int32)
    best = np.full(R, np.inf); second = np.full(R, np.inf)
    n_out = np.zeros(D, np.int32); m_out = np.zeros(D, np.int64)
    counts = np.zeros(3, np.int64)
    mi = None if m_init is None else _c(m_init, np.int64)
    ni = None if n_init is None else _c(n_init, np.int32)
    h = None if hint is None else _c(hint, np.int32)
    lib().oracle_schedule_stream_load(
        _p(f), _p(ro), _p(b), _p(la), _p(u), u.shape[1], _p(ln), _p(pf), _p(sn), _p(mm), _p(ev),
        len(ev), float(w_net), float(w_prefix), float(w_load), int(bytes_per_token), float(t_a),
        float(t_b), int(beta_max), int(m_min), int(m0), _p(mi), _p(ni), _p(h), float(rel_tol),
        _p(dec), _p(best), _p(second), _p(n_out), _p(m_out), _p(counts))
    return LoadResult(dec, best, second, n_out, m_out, int(counts[0]), int(counts[1]),
                      int(counts[2]))


UNBOUNDED = (1 << 64) - 1  # cache capacity that never evicts


class EvolvingResult(StreamResult):
    def __init__(self, dec, best, second, load, M, near_ties, mismatches, rejects, caches):
        super().__init__(dec, best, second, load, near_ties, mismatches, rejects)
        self.M = M
        self.caches = caches  # per decode: final cache, most recently used block first


def schedule_stream_evolving(fanout, role, bw, lat, util, length, prefill, snap, keys, key_off,
                             chains, chain_off, events, w_net, w_prefix, w_load, theta, cap,
                             bytes_per_token, hint=None, rel_tol=1e-5,
                             cap_blocks=UNBOUNDED) -> EvolvingResult:
    """Algorithm 1 with evolving caches, the simulator's LRU-managed block caches (Sec. VI-B):
    keys/key_off [D+1] are the decodes' caches at the stream's start, each list most
    recently used block first; a dispatch makes the request's chain the most recently used
    blocks of its decode's cache (block 0 the most recent) and evicts least recently used
    blocks beyond cap_blocks; M is taken per arrival against the caches of that moment and
    returned (.M), the final caches as lists (.caches)."""
    f, ro = _c(fanout, np.uint32), _c(role, np.uint8)
    b, la = _c(bw, np.float64), _c(lat, np.float64)
    u = _c(util, np.float32)
    ln, pf, sn = _c(length, np.uint32), _c(prefill, np.uint32), _c(snap, np.uint32)
    k, ko = _c(keys, np.uint64), _c(key_off, np.uint64)
    ch, co = _c(chains, np.uint64), _c(chain_off, np.uint64)
    ev = _c(events, np.uint32)
    R = len(ln)
    D = int((ro == 1).sum())
    assert len(ko) == D + 1 and len(co) == R + 1
    dec = np.full(R, -1, np.int32)
    best = np.full(R, np.inf); second = np.full(R, np.inf)
    M = np.zeros((R, D), np.uint16)
    load = np.zeros(D, np.int64)
    counts = np.zeros(3, np.int64)
    h = None if hint is None else _c(hint, np.int32)
    # room for the final caches: at most cap_blocks, or every key the stream ever saw
    stride = int(min(int(cap_blocks), len(k) + len(ch))) if D else 0
    stride = max(stride, 1)
    cache_out = np.zeros((D, stride), np.uint64)
    cache_len = np.zeros(D, np.uint64)
    lib().oracle_schedule_stream_evolving(
        _p(f), _p(ro), _p(b), _p(la), _p(u), u.shape[1], _p(ln), _p(pf), _p(sn), _p(k), _p(ko),
        int(cap_blocks), _p(ch), _p(co), _p(ev), len(ev), float(w_net), float(w_prefix),
        float(w_load), float(theta), int(cap), int(bytes_per_token), _p(h), float(rel_tol),
        _p(dec), _p(best), _p(second), _p(M), _p(load), _p(counts), _p(cache_out), stride,
        _p(cache_len))
    caches = [cache_out[d, :int(cache_len[d])].copy() for d in range(D)]
    return EvolvingResult(dec, best, second, load, M, int(counts[0]), int(counts[1]),
                          int(counts[2]), caches)
