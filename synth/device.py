"""Device materialisation of generated inputs (chains, cache keys, utilisations).

Large workloads do not fit a host-side generation pass, so the bulk arrays are
expanded on the GPU by ``synth_dev.cu`` from per-row keys computed here; the
values are identical to the host generator's (``synth.Workload.chains/keys/util``).
Small arrays (per-request attributes, events, offsets) come from the host.
"""
from __future__ import annotations

import ctypes as C
import os
import shutil
import subprocess
from typing import Optional

import numpy as np

from . import (DOWN_SEED, GOLDEN, MASK64, P_FILLER, P_ROOTHASH, P_TAIL, P_UTIL, Workload, _mix, stream_key,
               U64)

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "synth_dev.cu")
_LIB = os.path.join(_HERE, "libnetkv_synth.so")
_lib = None


def build(force: bool = False) -> str:
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O3",
                               "-Xcompiler", "-fPIC", "-shared", _SRC, "-o", tmp])
        os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB):
            build()
        _lib = C.CDLL(_LIB)
        P = C.c_void_p
        _lib.synth_chains.argtypes = [P, P, P, P, P, C.c_uint64, P]
        _lib.synth_keys.argtypes = [P, C.c_uint64, C.c_uint32, C.c_uint64, P, P, P]
        _lib.synth_util_uniform09.argtypes = [P, C.c_uint64, C.c_uint32, P, P]
        for f in ("synth_chains", "synth_keys", "synth_util_uniform09"):
            getattr(_lib, f).restype = C.c_int
    return _lib


def row_keys(seed_per_row: np.ndarray, purpose: int, a: np.ndarray) -> np.ndarray:
    """mix(stream_key(seed, purpose) + (a + 1) * GOLDEN) for each row."""
    seed_per_row = np.asarray(seed_per_row, dtype=np.int64)
    a = np.asarray(a, dtype=np.int64)
    seeds, inv = np.unique(seed_per_row, return_inverse=True)
    k = np.array([stream_key(int(s), purpose) for s in seeds], dtype=U64)
    with np.errstate(over="ignore"):
        return _mix(k[inv.reshape(-1)] + (a.astype(U64) + U64(1)) * U64(GOLDEN))


def _stream_ptr(stream) -> Optional[int]:
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return int(s.cuda_stream)


def _check(code, what):
    if code != 0:
        raise RuntimeError(f"{what} failed to launch ({code})")


def request_row_keys(w: Workload, r0: int, r1: int):
    r = np.arange(r0, r1, dtype=np.int64)
    s = np.searchsorted(w.req_off, r, side="right") - 1
    local = r - w.req_off[s]
    from . import request_set
    g = request_set(w)[r0:r1]
    rk = row_keys(w.set_seed[g], P_ROOTHASH, w.root[r0:r1].astype(np.int64))
    tk = row_keys(w.stream_seed[s], P_TAIL, local)
    return rk, tk


def chains(w: Workload, r0: int = 0, r1: Optional[int] = None, device="cuda", stream=None):
    """Chains of requests [r0, r1) as a device uint64 tensor, plus their offsets (from 0)."""
    import torch
    r1 = w.R if r1 is None else r1
    off = (w.chain_off[r0:r1 + 1] - w.chain_off[r0]).astype(np.uint64)
    rk, tk = request_row_keys(w, r0, r1)
    d_off = torch.from_numpy(off.view(np.int64)).to(device)
    d_rk = torch.from_numpy(rk.view(np.int64)).to(device)
    d_tk = torch.from_numpy(tk.view(np.int64)).to(device)
    d_sh = torch.from_numpy(w.shared[r0:r1].astype(np.int32)).to(device)
    out = torch.empty(int(off[-1]) if len(off) else 0, dtype=torch.int64, device=device)
    _check(lib().synth_chains(out.data_ptr(), d_off.data_ptr(), d_rk.data_ptr(), d_tk.data_ptr(),
                              d_sh.data_ptr(), r1 - r0, _stream_ptr(stream)), "synth_chains")
    return out, d_off


def key_segments(w: Workload, g0: int, g1: int):
    """Per-table segment row keys and cumulative bounds for table sets [g0, g1)."""
    spec = w.spec
    n_seg = spec.n_roots + 1
    T = (g1 - g0) * w.D
    seg_key = np.empty((T, n_seg), U64)
    cum = np.zeros((T, n_seg + 1), U64)
    kk = np.arange(spec.n_roots, dtype=np.int64)
    for gi, g in enumerate(range(g0, g1)):
        rk = row_keys(np.full(spec.n_roots, w.set_seed[g]), P_ROOTHASH, kk)
        fk = row_keys(np.full(w.D, w.set_seed[g]), P_FILLER, np.arange(w.D, dtype=np.int64))
        rows = slice(gi * w.D, (gi + 1) * w.D)
        seg_key[rows, :spec.n_roots] = rk[None, :]
        seg_key[rows, spec.n_roots] = fk
        depth = w.depth[g].astype(np.uint64)
        cum[rows, 1:spec.n_roots + 1] = np.cumsum(depth, axis=1)
        cum[rows, n_seg] = spec.n_keys
    return seg_key, cum


def keys(w: Workload, g0: int = 0, g1: Optional[int] = None, device="cuda", stream=None):
    """Cache key lists of table sets [g0, g1) as a device tensor [(g1-g0)*D*n_keys]."""
    import torch
    g1 = w.n_sets if g1 is None else g1
    seg_key, cum = key_segments(w, g0, g1)
    T = seg_key.shape[0]
    d_sk = torch.from_numpy(seg_key.reshape(-1).view(np.int64)).to(device)
    d_cum = torch.from_numpy(cum.reshape(-1).view(np.int64)).to(device)
    out = torch.empty(T * w.spec.n_keys, dtype=torch.int64, device=device)
    _check(lib().synth_keys(out.data_ptr(), T, seg_key.shape[1], w.spec.n_keys, d_sk.data_ptr(),
                            d_cum.data_ptr(), _stream_ptr(stream)), "synth_keys")
    return out


def util(w: Workload, s0: int = 0, s1: Optional[int] = None, device="cuda", stream=None,
         direction: str = "up"):
    """Utilisation rows [s0, s1) as a device fp32 tensor [s1-s0, L] (uniform modes on the
    device; Beta rows are generated on the host and copied).  direction as for
    synth.utilisation."""
    import torch
    s1 = w.n_snap if s1 is None else s1
    if w.spec.util_mode != "uniform09":
        return torch.from_numpy(w.util(s0, s1, direction)).to(device)
    shift = 0 if direction == "up" else DOWN_SEED
    rk = row_keys(w.snap_seed[s0:s1] + shift, P_UTIL, w.snap_local[s0:s1])
    d_rk = torch.from_numpy(rk.view(np.int64)).to(device)
    out = torch.empty((s1 - s0, w.L), dtype=torch.float32, device=device)
    _check(lib().synth_util_uniform09(out.data_ptr(), s1 - s0, w.L, d_rk.data_ptr(),
                                      _stream_ptr(stream)), "synth_util_uniform09")
    return out
