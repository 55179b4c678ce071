"""One step of the NetKV scoring path through the C ABI.

``Scorer`` holds what stays resident between steps (the topology handle and the
decode caches as an inverted hash index) and runs a step as three library calls on one
CUDA stream:

1. ``netkv_oracle_build``  -> level bottlenecks UB of every telemetry snapshot
2. ``netkv_prefix_match``  -> M[r][d] for every request and decode (with a
   workspace, so that requests sharing a prefix share the probing)
3. ``netkv_schedule_streams`` -> decisions, best/second scores, final loads
   (``netkv_schedule_streams_inflight`` when ``inflight_cap`` > 0: self-contention)

With evolving caches (``lru_setup``), steps 2 and 3 are one call,
``netkv_schedule_streams_evolving``: prefix hits are taken inside the greedy against
LRU-managed caches that every dispatch updates (``lru_reset`` sets them from key lists).

``step_host`` is the same step from host buffers: it copies the step's inputs
host->device (``netkv_copy_async``: SM-driven reads of pinned host memory), runs
the step and copies the results back, all on the stream.
Python here only marshals arguments; PyTorch provides device memory.
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import numpy as np
import torch

from . import netkv


@dataclasses.dataclass
class StepInputs:
    util: torch.Tensor        # f32 [n_snap, n_links]
    chains: torch.Tensor      # i64 (uint64 bits) [total blocks]
    chain_off: torch.Tensor   # i64 [R+1]
    set_off: torch.Tensor     # i32 [n_sets+1]
    length: torch.Tensor      # i32 [R]
    prefill: torch.Tensor     # i32 [R]
    snap: torch.Tensor        # i32 [R]
    events: torch.Tensor      # i32 (uint32 bits) [E]
    event_off: torch.Tensor   # i64 [n_streams+1]
    weights: torch.Tensor     # u8 [n_streams * 32] (netkv_weights)
    load_init: Optional[torch.Tensor] = None
    arrival_us: Optional[torch.Tensor] = None  # i64 [R], for self-contention
    util_down: Optional[torch.Tensor] = None   # f32 [n_snap, n_links], directed links

    @property
    def R(self) -> int:
        return int(self.length.shape[0])

    @property
    def n_streams(self) -> int:
        return int(self.event_off.shape[0] - 1)

    @property
    def n_snap(self) -> int:
        return int(self.util.shape[0])

    def nbytes(self) -> int:
        return sum(int(t.numel() * t.element_size()) for t in dataclasses.astuple(self)
                   if isinstance(t, torch.Tensor))


@dataclasses.dataclass
class StepOutputs:
    UB: torch.Tensor          # f32 [n_snap, N, 4]
    M: torch.Tensor           # i16 (uint16 bits) [R, D]
    dec: torch.Tensor         # i32 [R]
    best: torch.Tensor        # f32 [R]
    second: torch.Tensor      # f32 [R]
    load_final: torch.Tensor  # i64 [n_streams, D]
    status: torch.Tensor      # i32 [1]
    xfer_us: Optional[torch.Tensor] = None  # i32 [R], with self-contention
    held_final: Optional[torch.Tensor] = None  # i32 [n_streams, D], with the load model


class Scorer:
    def __init__(self, fanout, role, tier_bw, tier_lat, n_links: int, n_sets: int,
                 log2_capacity: int, device="cuda", share_prefixes: bool = True,
                 index: bool = True):
        """log2_capacity: slots per cache-index table (one table per table set and group
        of 64 decodes); see netkv.index_log2_capacity.  index=False: no static cache index
        (a scorer of evolving caches only)."""
        self.device = torch.device(device)
        self.topo = netkv.netkv_topology_create(fanout, role, tier_bw, tier_lat, n_links)
        self.N, self.P, self.D, self.used_links = netkv.netkv_topology_query(self.topo)
        self.n_links = int(n_links)
        self.n_sets = int(n_sets)
        self.log2_capacity = int(log2_capacity)
        nbytes = netkv.netkv_cache_index_bytes(self.n_sets, self.D, self.log2_capacity)
        self.index = (torch.empty(nbytes // 8, dtype=torch.int64, device=self.device) if index
                      else None)
        self.status = torch.zeros(1, dtype=torch.int32, device=self.device)
        self.share_prefixes = share_prefixes
        self.workspace = None
        self.precompute_scores = True
        self.sched_workspace = None
        # self-contention counter cap (Eq. 4's n_inflight); 0 = the plain greedy
        self.inflight_cap = 0
        # "links": per-link utilisation rows; "tiers": the paper's per-tier maps, x.util
        # then holds four congestion values per snapshot
        self.oracle_mode = "links"
        # the paper's compute-load model (netkv.LoadModel) instead of the token load;
        # out.load_final then holds free bytes and out.held_final request counts
        self.load_model = None
        # level bottlenecks from the utilisation rows inside the base-score pass
        # (netkv_schedule_streams_util): the step skips netkv_oracle_build and out.UB is
        # not written.  Used by the plain greedy with the base-score workspace only.
        self.fuse_level_bottlenecks = False
        # evolving LRU caches (netkv.LruConfig) and their state, one cache per
        # (stream, decode); None: the static caches of the index
        self.lru_cfg = None
        self.lru_state = None
        self.lru_caches = 0

    # ---- evolving caches
    def lru_setup(self, n_streams: int, cap_blocks: int) -> None:
        """State for the evolving caches of n_streams streams of cap_blocks blocks each."""
        self.lru_cfg = netkv.lru_config(cap_blocks)
        self.lru_caches = int(n_streams) * self.D
        nbytes = netkv.netkv_lru_state_bytes(self.lru_caches, self.lru_cfg)
        self.lru_state = torch.empty(nbytes // 8, dtype=torch.int64, device=self.device)

    def lru_reset(self, keys: torch.Tensor, key_off: torch.Tensor, stream=None,
                  n_caches: Optional[int] = None) -> None:
        """Every (stream, decode) cache from its key list, cache c = stream * D + decode,
        most recently used block first (the first n_caches caches when given)."""
        netkv.netkv_lru_init(self.lru_state, self.lru_caches if n_caches is None else n_caches,
                             self.lru_cfg, keys, key_off, self.status, stream)

    def lru_export(self, stream=None):
        """Each cache's blocks, most recently used first: (keys [caches, cap], lengths)."""
        cap = int(self.lru_cfg.cap_blocks)
        keys = torch.empty((self.lru_caches, cap), dtype=torch.int64, device=self.device)
        lens = torch.empty(self.lru_caches, dtype=torch.int64, device=self.device)
        netkv.netkv_lru_export(self.lru_state, self.lru_caches, self.lru_cfg, keys, lens,
                               self.status, stream)
        return keys, lens

    def _sched_workspace(self, R: int):
        """Greedy workspace (base scores of every arrival), grown on demand."""
        if not self.precompute_scores:
            return None
        need = netkv.netkv_schedule_workspace_size(R, self.D)
        if self.sched_workspace is None or self.sched_workspace.numel() < need:
            self.sched_workspace = torch.empty(max(need, 256), dtype=torch.uint8,
                                               device=self.device)
        return self.sched_workspace

    def _workspace(self, R: int):
        """Prefix-match workspace for R requests (grown on demand, reused across steps)."""
        if not self.share_prefixes:
            return None
        need = netkv.netkv_prefix_match_workspace_size(R)
        if self.workspace is None or self.workspace.numel() < need:
            self.workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=self.device)
        return self.workspace

    # ---- resident state
    def load_caches(self, keys: torch.Tensor, key_off: torch.Tensor, set0: int = 0,
                    n_sets: Optional[int] = None, stream=None) -> None:
        """Build the tables of table sets [set0, set0 + n_sets) from a key list."""
        n_sets = self.n_sets - set0 if n_sets is None else n_sets
        off = netkv.netkv_cache_index_bytes(set0, self.D, self.log2_capacity) // 8
        netkv.netkv_cache_build(self.index[off:], n_sets, self.D, self.log2_capacity, keys,
                                key_off, self.status, stream)

    # ---- one step
    def alloc_outputs(self, n_snap: int, R: int, n_streams: int) -> StepOutputs:
        dev = self.device
        return StepOutputs(
            UB=torch.empty((n_snap, self.N, 4), dtype=torch.float32, device=dev),
            M=torch.empty((R, self.D), dtype=torch.int16, device=dev),
            dec=torch.empty(R, dtype=torch.int32, device=dev),
            best=torch.empty(R, dtype=torch.float32, device=dev),
            second=torch.empty(R, dtype=torch.float32, device=dev),
            load_final=torch.empty((n_streams, self.D), dtype=torch.int64, device=dev),
            status=torch.zeros(1, dtype=torch.int32, device=dev),
            xfer_us=torch.empty(R, dtype=torch.int32, device=dev),
            held_final=torch.empty((n_streams, self.D), dtype=torch.int32, device=dev))

    def oracle_build(self, x: StepInputs, out: StepOutputs, stream=None) -> None:
        if self.oracle_mode == "tiers":
            netkv.netkv_oracle_build_tiers(self.topo, x.util, x.n_snap, 1.0, None, out.UB,
                                           out.status, stream)
            return
        if x.util_down is not None:  # directed links: util holds the upward rows
            netkv.netkv_oracle_build_directed(self.topo, x.util, x.util_down, x.n_snap, 1.0, None,
                                              out.UB, out.status, stream)
            return
        netkv.netkv_oracle_build(self.topo, x.util, x.n_snap, 1.0, None, out.UB, out.status, stream)

    def schedule_evolving(self, x: StepInputs, out: StepOutputs, stream=None, streams=None) -> None:
        """Prefix hits and the greedy in one call, against the evolving caches; streams =
        (j0, j1) runs streams j0 .. j1-1 on the caches of the state's first j1 - j0 streams."""
        j0, j1 = (0, x.n_streams) if streams is None else streams
        netkv.netkv_schedule_streams_evolving(
            self.topo, j1 - j0, x.weights[32 * j0:], x.R, x.length, x.prefill, x.snap, out.UB,
            x.n_snap, x.chains, x.chain_off, x.events, x.event_off[j0:], self.lru_state,
            self.lru_cfg, None if x.load_init is None else x.load_init[j0:], out.dec, out.best,
            out.second, out.M, out.load_final[j0:], out.status, stream)

    def prefix_match(self, x: StepInputs, out: StepOutputs, stream=None) -> None:
        netkv.netkv_prefix_match(self.index, self.D, self.log2_capacity, self.n_sets, x.chains,
                                 x.chain_off, x.R, x.set_off if self.n_sets > 1 else None, out.M,
                                 out.status, stream, workspace=self._workspace(x.R))

    def schedule(self, x: StepInputs, out: StepOutputs, stream=None) -> None:
        if self.load_model is not None:
            netkv.netkv_schedule_streams_load(
                self.topo, x.n_streams, x.weights, self.load_model, x.R, x.length, x.prefill,
                x.snap, out.M, out.UB, x.n_snap, x.events, x.event_off, None, None, out.dec,
                out.best, out.second, out.load_final, out.held_final, out.status, stream)
            return
        if self.inflight_cap > 0:
            netkv.netkv_schedule_streams_inflight(
                self.topo, x.n_streams, x.weights, x.R, x.length, x.prefill, x.snap,
                x.arrival_us, out.M, out.UB, x.n_snap, x.events, x.event_off, self.inflight_cap,
                x.load_init, out.dec, out.best, out.second, out.xfer_us, out.load_final,
                out.status, stream)  # the walk, not its scoring, bounds this form
            return
        if self.fused(x):
            netkv.netkv_schedule_streams_util(
                self.topo, x.n_streams, x.weights, x.R, x.length, x.prefill, x.snap, out.M,
                x.util, x.n_snap, x.events, x.event_off, x.load_init, out.dec, out.best,
                out.second, out.load_final, out.status, stream,
                workspace=self._sched_workspace(x.R))
            return
        netkv.netkv_schedule_streams(self.topo, x.n_streams, x.weights, x.R, x.length, x.prefill,
                                     x.snap, out.M, out.UB, x.n_snap, x.events, x.event_off,
                                     x.load_init, out.dec, out.best, out.second, out.load_final,
                                     out.status, stream, workspace=self._sched_workspace(x.R))

    def fused(self, x: StepInputs) -> bool:
        """Whether the step takes the level bottlenecks from the utilisation rows."""
        return (self.fuse_level_bottlenecks and self.precompute_scores and
                self.oracle_mode == "links" and x.util_down is None and self.inflight_cap == 0
                and self.load_model is None and self.lru_cfg is None)

    def step(self, x: StepInputs, out: StepOutputs, stream=None) -> StepOutputs:
        if self.fused(x):
            self.prefix_match(x, out, stream)
            self.schedule(x, out, stream)
            return out
        self.oracle_build(x, out, stream)
        if self.lru_cfg is not None:
            self.schedule_evolving(x, out, stream)
            return out
        self.prefix_match(x, out, stream)
        self.schedule(x, out, stream)
        return out

    def step_host(self, xh: StepInputs, xd: StepInputs, out: StepOutputs, res_h: dict,
                  stream=None, zero_copy=()) -> StepOutputs:
        """Host-buffer step: xh holds pinned host tensors, xd same-shaped device tensors,
        res_h pinned host tensors for dec/best/second/load_final.

        Fields named in `zero_copy` are not copied: the kernels read them in place from
        pinned host memory (unified addressing over NVLink-C2C), so only the parts a step
        actually touches cross the link (for the chains: blocks up to each first miss)."""
        s = torch.cuda.current_stream() if stream is None else stream
        for f in dataclasses.fields(StepInputs):
            h = getattr(xh, f.name)
            if isinstance(h, torch.Tensor) and f.name not in zero_copy:
                d = getattr(xd, f.name)
                netkv.netkv_copy_async(d, h, h.numel() * h.element_size(), s)
        if zero_copy:
            xd = dataclasses.replace(xd, **{name: getattr(xh, name) for name in zero_copy})
        self.step(xd, out, s)
        for k in ("dec", "best", "second", "load_final"):
            d = getattr(out, k)
            netkv.netkv_copy_async(res_h[k], d, d.numel() * d.element_size(), s)
        return out


def weights_tensor(w: np.ndarray, theta: float, cap_tokens: int, bytes_per_token: int,
                   device="cuda") -> torch.Tensor:
    host = netkv.make_weights(w, theta, cap_tokens, bytes_per_token)
    return torch.from_numpy(host.view(np.uint8).copy()).to(device)
