"""Stage a generated workload on the device (inputs only; no scoring arithmetic).

Returns plain dicts of torch tensors: per-request arrays, offsets, events and
the bulk arrays (chains, cache key lists, utilisations), the bulk ones expanded
on the GPU by ``synth.device``.  Unsigned values are carried in signed tensors
of the same width (torch has no uint32/uint64 arithmetic needs here).
"""
from __future__ import annotations

from typing import Dict, Optional

import numpy as np

from . import Workload
from . import device as sdev


def _t(a: np.ndarray, dtype, device):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a).view(dtype)).to(device)


def request_arrays(w: Workload, device="cuda", pin: bool = False) -> Dict[str, "torch.Tensor"]:
    """Per-step request inputs, on `device` (or pinned host memory when device='cpu', pin)."""
    import torch
    d = {
        "chain_off": w.chain_off.astype(np.uint64).view(np.int64),
        "set_off": w.set_off.astype(np.uint32).view(np.int32),
        "length": w.length.astype(np.uint32).view(np.int32),
        "prefill": w.prefill.astype(np.uint32).view(np.int32),
        "snap": w.snap.astype(np.uint32).view(np.int32),
        "events": w.events.astype(np.uint32).view(np.int32),
        "event_off": w.event_off.astype(np.uint64).view(np.int64),
    }
    out = {}
    for k, v in d.items():
        t = torch.from_numpy(np.ascontiguousarray(v))
        out[k] = t.pin_memory() if (pin and device == "cpu") else t.to(device)
    return out


def key_offsets(w: Workload, n_tables: int, device="cuda"):
    import torch
    off = (np.arange(n_tables + 1, dtype=np.int64) * w.spec.n_keys)
    return torch.from_numpy(off).to(device)


def chains(w: Workload, device="cuda", host_threshold: int = 1 << 22):
    """All chains as a device tensor (host generation for small workloads)."""
    import torch
    total = int(w.chain_off[-1])
    if total <= host_threshold:
        return torch.from_numpy(w.chains().view(np.int64)).to(device)
    return sdev.chains(w, device=device)[0]


def keys(w: Workload, g0: int, g1: int, device="cuda", host_threshold: int = 1 << 22):
    import torch
    if (g1 - g0) * w.D * w.spec.n_keys <= host_threshold:
        ks = [w.keys(g, d) for g in range(g0, g1) for d in range(w.D)]
        return torch.from_numpy(np.concatenate(ks).view(np.int64)).to(device)
    return sdev.keys(w, g0, g1, device=device)


def util(w: Workload, device="cuda", host_threshold: int = 1 << 22, direction: str = "up"):
    import torch
    if direction == "tiers" or w.n_snap * w.L <= host_threshold or w.spec.util_mode != "uniform09":
        return torch.from_numpy(w.util(direction=direction)).to(device)
    return sdev.util(w, device=device, direction=direction)
