"""Thin Python binding of the NetKV C ABI (``include/netkv.h``).

Argument marshalling only: every function forwards to the entry point of the
same name in ``libnetkv.so``; all computation happens in the CUDA kernels
behind it.  Device buffers may be given as torch tensors (their ``data_ptr()``
is passed) or as raw integer device addresses; ``None`` passes NULL.  A
non-OK status raises :class:`NetKVError`.  There is no CPU fallback: if the
library is missing, importing this module fails.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libnetkv.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: build it first "
                      "(python -c 'import __graft_entry__ as g; g.build()')")
_lib = C.CDLL(LIB_PATH)

NETKV_OK, NETKV_EINVAL, NETKV_ENOMEM, NETKV_ECUDA, NETKV_ELIMIT = 0, 1, 2, 3, 4
NETKV_PREFIX_MATCH_STATIC_MAX_R = 524288
NETKV_DEV_EDOMAIN, NETKV_DEV_EFULL, NETKV_DEV_ERANGE = 1, 2, 4
_NAMES = {1: "NETKV_EINVAL", 2: "NETKV_ENOMEM", 3: "NETKV_ECUDA",
          4: "NETKV_ELIMIT (more requests than the fixed scratch of netkv_prefix_match_static holds)"}

EXPORTS = ("netkv_topology_create", "netkv_topology_destroy", "netkv_topology_query",
           "netkv_oracle_build", "netkv_oracle_build_directed", "netkv_oracle_build_tiers",
           "netkv_cache_index_bytes",
           "netkv_cache_build",
           "netkv_prefix_match_workspace_size",
           "netkv_prefix_match", "netkv_prefix_match_static", "netkv_schedule_workspace_size",
           "netkv_schedule_streams", "netkv_schedule_streams_util",
           "netkv_schedule_streams_inflight",
           "netkv_schedule_inflight_workspace_size",
           "netkv_schedule_streams_load",
           "netkv_lru_state_bytes", "netkv_lru_init", "netkv_lru_export",
           "netkv_schedule_streams_evolving",
           "netkv_copy_async", "netkv_version")


class NetKVError(RuntimeError):
    def __init__(self, fn: str, code: int):
        super().__init__(f"{fn} returned {_NAMES.get(code, code)}")
        self.code = code


class _Desc(C.Structure):
    _fields_ = [("fanout", C.c_uint32 * 4), ("role", C.c_void_p),
                ("tier_bw_Bps", C.c_double * 4), ("tier_lat_s", C.c_double * 4),
                ("n_links", C.c_uint32)]


# netkv_weights, 32 bytes: 4 x f32, i64, u64
WEIGHTS_DTYPE = np.dtype([("w_net", "<f4"), ("w_prefix", "<f4"), ("w_load", "<f4"),
                          ("theta_s_per_token", "<f4"), ("cap_tokens", "<i8"),
                          ("bytes_per_token", "<u8")])
assert WEIGHTS_DTYPE.itemsize == 32

_P, _U32, _U64, _F64 = C.c_void_p, C.c_uint32, C.c_uint64, C.c_double
_lib.netkv_version.restype = C.c_uint32
_lib.netkv_topology_create.argtypes = [C.POINTER(_Desc), C.POINTER(C.c_void_p)]
_lib.netkv_topology_destroy.argtypes = [_P]
_lib.netkv_topology_query.argtypes = [_P, _P, _P, _P, _P]
_lib.netkv_oracle_build.argtypes = [_P, _P, _U32, _F64, _P, _P, _P, _P]
_lib.netkv_oracle_build_directed.argtypes = [_P, _P, _P, _U32, _F64, _P, _P, _P, _P]
_lib.netkv_oracle_build_tiers.argtypes = [_P, _P, _U32, _F64, _P, _P, _P, _P]
_lib.netkv_cache_index_bytes.argtypes = [_U32, _U32, _U32]
_lib.netkv_cache_index_bytes.restype = C.c_size_t
_lib.netkv_cache_build.argtypes = [_P, _U32, _U32, _U32, _P, _P, _P, _P]
_lib.netkv_prefix_match_workspace_size.argtypes = [_U32]
_lib.netkv_prefix_match_workspace_size.restype = C.c_size_t
_lib.netkv_prefix_match.argtypes = [_P, _U32, _U32, _U32, _P, _P, _U32, _P, _P, C.c_size_t, _P,
                                    _P, _P]
_lib.netkv_prefix_match_static.argtypes = [_P, _U32, _U32, _U32, _P, _P, _U32, _P, _P, _P, _P]
_lib.netkv_schedule_workspace_size.argtypes = [_U32, _U32]
_lib.netkv_schedule_workspace_size.restype = C.c_size_t
_lib.netkv_schedule_streams.argtypes = [_P, _U32, _P, _U32, _P, _P, _P, _P, _P, _U32, _P, _P,
                                        _P, _P, _P, _P, _P, _P, C.c_size_t, _P, _P]
_lib.netkv_schedule_streams_util.argtypes = [_P, _U32, _P, _U32, _P, _P, _P, _P, _P, _U32, _P,
                                             _P, _P, _P, _P, _P, _P, _P, C.c_size_t, _P, _P]
_lib.netkv_schedule_streams_inflight.argtypes = [_P, _U32, _P, _U32, _P, _P, _P, _P, _P, _P,
                                                 _U32, _P, _P, _U32, _P, _P, _P, _P, _P, _P,
                                                 _P, C.c_size_t, _P, _P]
_lib.netkv_schedule_inflight_workspace_size.argtypes = [_U32, _U32]
_lib.netkv_schedule_inflight_workspace_size.restype = C.c_size_t
class LoadModel(C.Structure):
    """netkv_load_model: the paper's compute-load model constants (Sec. III-C, IV-B)."""
    _fields_ = [("t_a_s", C.c_float), ("t_b_s", C.c_float), ("beta_max", C.c_int32),
                ("reserved", C.c_int32), ("m_min_bytes", C.c_int64), ("m0_bytes", C.c_int64)]


_lib.netkv_schedule_streams_load.argtypes = [_P, _U32, _P, C.POINTER(LoadModel), _U32, _P, _P,
                                             _P, _P, _P, _U32, _P, _P, _P, _P, _P, _P, _P, _P,
                                             _P, _P, _P]
class LruConfig(C.Structure):
    """netkv_lru_config: capacity and table sizes of the evolving (LRU) decode caches."""
    _fields_ = [("cap_blocks", C.c_uint64), ("log2_slots", C.c_uint32), ("log2_ring", C.c_uint32)]


def lru_config(cap_blocks: int) -> LruConfig:
    """The smallest tables netkv.h allows for caches of cap_blocks blocks."""
    need = int(cap_blocks) + 65536
    ls = 4
    while (3 << ls) // 4 < need - 1:
        ls += 1
    lr = 4
    while (1 << lr) < need:
        lr += 1
    return LruConfig(int(cap_blocks), ls, lr)


_lib.netkv_lru_state_bytes.argtypes = [_U64, C.POINTER(LruConfig)]
_lib.netkv_lru_state_bytes.restype = C.c_size_t
_lib.netkv_lru_init.argtypes = [_P, C.c_size_t, _U64, C.POINTER(LruConfig), _P, _P, _P, _P]
_lib.netkv_lru_export.argtypes = [_P, C.c_size_t, _U64, C.POINTER(LruConfig), _P, _P, _P, _P]
_lib.netkv_schedule_streams_evolving.argtypes = [_P, _U32, _P, _U32, _P, _P, _P, _P, _U32, _P, _P,
                                                 _P, _P, _P, C.c_size_t, C.POINTER(LruConfig), _P,
                                                 _P, _P, _P, _P, _P, _P, _P]
_lib.netkv_copy_async.argtypes = [_P, _P, C.c_size_t, _P]
for _f in EXPORTS:
    if _f not in ("netkv_version", "netkv_prefix_match_workspace_size", "netkv_cache_index_bytes",
                  "netkv_schedule_workspace_size", "netkv_schedule_inflight_workspace_size",
                  "netkv_lru_state_bytes"):
        getattr(_lib, _f).restype = C.c_int


def _ptr(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return int(x.data_ptr())


def _stream(s) -> Optional[int]:
    if s is None:
        import torch
        return int(torch.cuda.current_stream().cuda_stream) if torch.cuda.is_initialized() else None
    if isinstance(s, int):
        return s
    return int(s.cuda_stream)


def _check(fn: str, code: int) -> None:
    if code != NETKV_OK:
        raise NetKVError(fn, code)


def netkv_version() -> int:
    return int(_lib.netkv_version())


class Topology:
    """Owns a netkv_topology_t handle (released by netkv_topology_destroy)."""

    def __init__(self, handle: int):
        self.handle = handle

    @property
    def as_parameter(self):
        return self.handle

    def __del__(self):
        if getattr(self, "handle", None):
            try:
                _lib.netkv_topology_destroy(self.handle)
            except Exception:
                pass
            self.handle = None


def netkv_topology_create(fanout: Sequence[int], role: np.ndarray, tier_bw_Bps: Sequence[float],
                          tier_lat_s: Sequence[float], n_links: int) -> Topology:
    role = np.ascontiguousarray(role, dtype=np.uint8)
    d = _Desc()
    d.fanout[:] = [int(x) for x in fanout]
    d.role = role.ctypes.data
    d.tier_bw_Bps[:] = [float(x) for x in tier_bw_Bps]
    d.tier_lat_s[:] = [float(x) for x in tier_lat_s]
    d.n_links = int(n_links)
    h = C.c_void_p()
    _check("netkv_topology_create", _lib.netkv_topology_create(C.byref(d), C.byref(h)))
    return Topology(h.value)


def netkv_topology_destroy(topo: Topology) -> None:
    if topo.handle:
        _check("netkv_topology_destroy", _lib.netkv_topology_destroy(topo.handle))
        topo.handle = None


def netkv_topology_query(topo: Topology):
    v = [C.c_uint32() for _ in range(4)]
    _check("netkv_topology_query",
           _lib.netkv_topology_query(topo.handle, *[C.byref(x) for x in v]))
    return tuple(int(x.value) for x in v)


def netkv_oracle_build(topo: Topology, util, n_snap: int, kv_bytes: float, C_out=None, UB=None,
                       status=None, stream=None) -> None:
    _check("netkv_oracle_build", _lib.netkv_oracle_build(
        topo.handle, _ptr(util), int(n_snap), float(kv_bytes), _ptr(C_out), _ptr(UB),
        _ptr(status), _stream(stream)))


def netkv_cache_index_bytes(n_sets: int, D: int, log2_capacity: int) -> int:
    return int(_lib.netkv_cache_index_bytes(int(n_sets), int(D), int(log2_capacity)))


def netkv_cache_build(index, n_sets: int, D: int, log2_capacity: int, keys, key_off, status=None,
                      stream=None) -> None:
    _check("netkv_cache_build", _lib.netkv_cache_build(
        _ptr(index), int(n_sets), int(D), int(log2_capacity), _ptr(keys), _ptr(key_off),
        _ptr(status), _stream(stream)))


def netkv_prefix_match_workspace_size(R: int) -> int:
    return int(_lib.netkv_prefix_match_workspace_size(int(R)))


def netkv_prefix_match(index, D: int, log2_capacity: int, n_sets: int, chains, chain_off, R: int,
                       set_off, M, status=None, stream=None, workspace=None) -> None:
    ws_bytes = 0 if workspace is None else int(workspace.numel() * workspace.element_size())
    _check("netkv_prefix_match", _lib.netkv_prefix_match(
        _ptr(index), int(D), int(log2_capacity), int(n_sets), _ptr(chains), _ptr(chain_off),
        int(R), _ptr(set_off), _ptr(workspace), ws_bytes, _ptr(M), _ptr(status), _stream(stream)))


def netkv_prefix_match_static(index, D: int, log2_capacity: int, n_sets: int, chains, chain_off,
                              R: int, set_off, M, status=None, stream=None) -> None:
    """Prefix match that allocates nothing (fixed device scratch inside the library);
    for callers that may not allocate device memory.  Overlapping calls race."""
    _check("netkv_prefix_match_static", _lib.netkv_prefix_match_static(
        _ptr(index), int(D), int(log2_capacity), int(n_sets), _ptr(chains), _ptr(chain_off),
        int(R), _ptr(set_off), _ptr(M), _ptr(status), _stream(stream)))


def netkv_schedule_workspace_size(R: int, D: int) -> int:
    return int(_lib.netkv_schedule_workspace_size(int(R), int(D)))


def netkv_schedule_streams(topo: Topology, n_streams: int, weights, R: int, length, prefill, snap,
                           M, UB, n_snap: int, events, event_off, load_init, dec, best, second,
                           load_final, status=None, stream=None, workspace=None) -> None:
    ws_bytes = 0 if workspace is None else int(workspace.numel() * workspace.element_size())
    _check("netkv_schedule_streams", _lib.netkv_schedule_streams(
        topo.handle, int(n_streams), _ptr(weights), int(R), _ptr(length), _ptr(prefill),
        _ptr(snap), _ptr(M), _ptr(UB), int(n_snap), _ptr(events), _ptr(event_off),
        _ptr(load_init), _ptr(dec), _ptr(best), _ptr(second), _ptr(load_final), _ptr(workspace),
        ws_bytes, _ptr(status), _stream(stream)))


def netkv_schedule_streams_util(topo: Topology, n_streams: int, weights, R: int, length, prefill,
                                snap, M, util, n_snap: int, events, event_off, load_init, dec,
                                best, second, load_final, status=None, stream=None,
                                workspace=None) -> None:
    """The greedy with level bottlenecks from the utilisation rows; see include/netkv.h."""
    ws_bytes = 0 if workspace is None else int(workspace.numel() * workspace.element_size())
    _check("netkv_schedule_streams_util", _lib.netkv_schedule_streams_util(
        topo.handle, int(n_streams), _ptr(weights), int(R), _ptr(length), _ptr(prefill),
        _ptr(snap), _ptr(M), _ptr(util), int(n_snap), _ptr(events), _ptr(event_off),
        _ptr(load_init), _ptr(dec), _ptr(best), _ptr(second), _ptr(load_final), _ptr(workspace),
        ws_bytes, _ptr(status), _stream(stream)))


def netkv_schedule_streams_inflight(topo: Topology, n_streams: int, weights, R: int, length,
                                    prefill, snap, arrival_us, M, UB, n_snap: int, events,
                                    event_off, inflight_cap: int, load_init, dec, best, second,
                                    xfer_us, load_final, status=None, stream=None,
                                    workspace=None) -> None:
    """Algorithm 1 with self-contention; see include/netkv.h."""
    ws_bytes = 0 if workspace is None else int(workspace.numel() * workspace.element_size())
    _check("netkv_schedule_streams_inflight", _lib.netkv_schedule_streams_inflight(
        topo.handle, int(n_streams), _ptr(weights), int(R), _ptr(length), _ptr(prefill),
        _ptr(snap), _ptr(arrival_us), _ptr(M), _ptr(UB), int(n_snap), _ptr(events),
        _ptr(event_off), int(inflight_cap), _ptr(load_init), _ptr(dec), _ptr(best),
        _ptr(second), _ptr(xfer_us), _ptr(load_final), _ptr(workspace), ws_bytes, _ptr(status),
        _stream(stream)))


def netkv_schedule_inflight_workspace_size(R: int, D: int) -> int:
    return int(_lib.netkv_schedule_inflight_workspace_size(int(R), int(D)))


def netkv_oracle_build_directed(topo: Topology, util_up, util_down, n_snap: int, kv_bytes: float,
                                C=None, UB=None, status=None, stream=None) -> None:
    """Oracle build with directed links; see include/netkv.h."""
    _check("netkv_oracle_build_directed", _lib.netkv_oracle_build_directed(
        topo.handle, _ptr(util_up), _ptr(util_down), int(n_snap), float(kv_bytes), _ptr(C),
        _ptr(UB), _ptr(status), _stream(stream)))


def netkv_oracle_build_tiers(topo: Topology, c, n_snap: int, kv_bytes: float, C=None, UB=None,
                             status=None, stream=None) -> None:
    """The paper-literal per-tier oracle; see include/netkv.h."""
    _check("netkv_oracle_build_tiers", _lib.netkv_oracle_build_tiers(
        topo.handle, _ptr(c), int(n_snap), float(kv_bytes), _ptr(C), _ptr(UB), _ptr(status),
        _stream(stream)))


def netkv_schedule_streams_load(topo: Topology, n_streams: int, weights, model: LoadModel, R: int,
                                length, prefill, snap, M, UB, n_snap: int, events, event_off,
                                m_init, n_init, dec, best, second, m_final, n_final,
                                status=None, stream=None) -> None:
    """Algorithm 1 with the paper's compute-load model; see include/netkv.h."""
    _check("netkv_schedule_streams_load", _lib.netkv_schedule_streams_load(
        topo.handle, int(n_streams), _ptr(weights), C.byref(model), int(R), _ptr(length),
        _ptr(prefill), _ptr(snap), _ptr(M), _ptr(UB), int(n_snap), _ptr(events), _ptr(event_off),
        _ptr(m_init), _ptr(n_init), _ptr(dec), _ptr(best), _ptr(second), _ptr(m_final),
        _ptr(n_final), _ptr(status), _stream(stream)))


def netkv_lru_state_bytes(n_caches: int, cfg: LruConfig) -> int:
    return int(_lib.netkv_lru_state_bytes(int(n_caches), C.byref(cfg)))


def _nbytes(t) -> int:
    return int(t.numel() * t.element_size())


def netkv_lru_init(state, n_caches: int, cfg: LruConfig, keys, key_off, status=None,
                   stream=None) -> None:
    """Evolving caches from key lists (most recently used first); see include/netkv.h."""
    _check("netkv_lru_init", _lib.netkv_lru_init(_ptr(state), _nbytes(state), int(n_caches),
                                                 C.byref(cfg), _ptr(keys), _ptr(key_off),
                                                 _ptr(status), _stream(stream)))


def netkv_lru_export(state, n_caches: int, cfg: LruConfig, keys_out, len_out, status=None,
                     stream=None) -> None:
    """Every evolving cache's blocks, most recently used first; see include/netkv.h."""
    _check("netkv_lru_export", _lib.netkv_lru_export(_ptr(state), _nbytes(state), int(n_caches),
                                                     C.byref(cfg), _ptr(keys_out), _ptr(len_out),
                                                     _ptr(status), _stream(stream)))


def netkv_schedule_streams_evolving(topo: Topology, n_streams: int, weights, R: int, length,
                                    prefill, snap, UB, n_snap: int, chains, chain_off, events,
                                    event_off, state, cfg: LruConfig, load_init, dec, best,
                                    second, M, load_final, status=None, stream=None) -> None:
    """Algorithm 1 with evolving LRU caches; see include/netkv.h."""
    _check("netkv_schedule_streams_evolving", _lib.netkv_schedule_streams_evolving(
        topo.handle, int(n_streams), _ptr(weights), int(R), _ptr(length), _ptr(prefill),
        _ptr(snap), _ptr(UB), int(n_snap), _ptr(chains), _ptr(chain_off), _ptr(events),
        _ptr(event_off), _ptr(state), _nbytes(state), C.byref(cfg), _ptr(load_init), _ptr(dec),
        _ptr(best),
        _ptr(second), _ptr(M), _ptr(load_final), _ptr(status), _stream(stream)))


def netkv_copy_async(dst, src, nbytes: int, stream=None) -> None:
    """Kernel copy between device and/or pinned host buffers (torch tensors or addresses)."""
    _check("netkv_copy_async", _lib.netkv_copy_async(_ptr(dst), _ptr(src), int(nbytes),
                                                     _stream(stream)))


def make_weights(w: np.ndarray, theta: float, cap_tokens: int, bytes_per_token: int) -> np.ndarray:
    """Host array of netkv_weights from an [n_streams, 3] (w_net, w_prefix, w_load) array."""
    w = np.asarray(w, dtype=np.float32).reshape(-1, 3)
    out = np.zeros(len(w), WEIGHTS_DTYPE)
    out["w_net"], out["w_prefix"], out["w_load"] = w[:, 0], w[:, 1], w[:, 2]
    out["theta_s_per_token"] = np.float32(theta)
    out["cap_tokens"] = int(cap_tokens)
    out["bytes_per_token"] = int(bytes_per_token)
    return out


def index_log2_capacity(max_distinct_keys: int) -> int:
    """Smallest table size keeping a cache-index table at load factor <= 0.5."""
    l = 1
    while (1 << l) < 2 * max(int(max_distinct_keys), 1):
        l += 1
    return l
