"""A second, deliberately naive evaluator used only to pin the C++ oracle.

It shares nothing with the oracle: the instance tree is built as an explicit
graph (named vertices, adjacency lists), paths come from breadth-first search,
prefix hits from a list scan, and scores are exact rationals (``fractions``),
so every comparison is free of rounding.  Only tiny instances are feasible.
"""
from __future__ import annotations

from collections import deque
from fractions import Fraction
from typing import Dict, List, Sequence, Tuple

import numpy as np


class ExplicitTree:
    """Vertices: ('inst', i), ('node', n), ('leaf', l), ('pod', q), ('spine',).

    Edge ids follow the link numbering of the library's interface: instance-node
    links first (by instance), then node-leaf links (by node), leaf-pod links (by
    leaf), pod-spine links (by pod).  Each edge also records its level 0..3.
    """

    def __init__(self, fanout: Sequence[int]):
        f0, f1, f2, f3 = fanout
        self.n = f0 * f1 * f2 * f3
        n_node, n_leaf, n_pod = self.n // f0, self.n // (f0 * f1), f3
        self.adj: Dict[tuple, List[Tuple[tuple, int]]] = {}
        self.level: Dict[int, int] = {}
        eid = 0

        def add(a, b, lvl):
            nonlocal eid
            self.adj.setdefault(a, []).append((b, eid))
            self.adj.setdefault(b, []).append((a, eid))
            self.level[eid] = lvl
            eid += 1

        for i in range(self.n):
            add(("inst", i), ("node", i // f0), 0)
        for nd in range(n_node):
            add(("node", nd), ("leaf", nd // f1), 1)
        for lf in range(n_leaf):
            add(("leaf", lf), ("pod", lf // f2), 2)
        for q in range(n_pod):
            add(("pod", q), ("spine",), 3)
        self.n_edges = eid

    def path(self, i: int, j: int) -> List[int]:
        src, dst = ("inst", i), ("inst", j)
        prev = {src: None}
        q = deque([src])
        while q:
            v = q.popleft()
            if v == dst:
                break
            for w, e in self.adj[v]:
                if w not in prev:
                    prev[w] = (v, e)
                    q.append(w)
        edges = []
        v = dst
        while prev[v] is not None:
            v, e = prev[v]
            edges.append(e)
        return edges[::-1]

    def path_steps(self, i: int, j: int) -> List[Tuple[int, bool]]:
        """(edge, climbing) along the path from instance i to instance j: climbing when the
        step goes from a vertex to one higher in the tree (instance < node < leaf < pod <
        spine)."""
        height = {"inst": 0, "node": 1, "leaf": 2, "pod": 3, "spine": 4}
        src, dst = ("inst", i), ("inst", j)
        prev = {src: None}
        q = deque([src])
        while q:
            v = q.popleft()
            if v == dst:
                break
            for w, e in self.adj[v]:
                if w not in prev:
                    prev[w] = (v, e)
                    q.append(w)
        steps = []
        v = dst
        while prev[v] is not None:
            u, e = prev[v]
            steps.append((e, height[v[0]] > height[u[0]]))
            v = u
        return steps[::-1]

    def tier(self, i: int, j: int) -> int:
        # the highest level among the path's edges is the tier of the pair
        return max(self.level[e] for e in self.path(i, j))


def frac(x) -> Fraction:
    return Fraction(float(x))


def bottleneck(tree: ExplicitTree, bw, u_row, i, j) -> Fraction:
    return min(frac(bw[tree.level[e]]) * (1 - frac(u_row[e])) for e in tree.path(i, j))


def bottleneck_directed(tree: ExplicitTree, bw, u_up_row, u_down_row, i, j) -> Fraction:
    """Directed links: each step of the path from i to j at the utilisation of the
    direction it crosses the link in."""
    return min(frac(bw[tree.level[e]]) * (1 - frac((u_up_row if up else u_down_row)[e]))
               for e, up in tree.path_steps(i, j))


def cost(tree, bw, lat, u_row, i, j, kv) -> Fraction:
    return frac(kv) / bottleneck(tree, bw, u_row, i, j) + frac(lat[tree.tier(i, j)])


def lcp_blocks(chain: Sequence[int], cache: Sequence[int]) -> int:
    m = 0
    for h in chain:
        if h not in cache:
            break
        m += 1
    return m


def greedy_exact(tree, role, bw, lat, util, length, prefill, snap, M, events,
                 w, theta, cap, bpt, util_down=None, tier_mode=False):
    """Exact-rational Algorithm 1 with the weighted score; returns (dec, best_scores).
    util_down: downward rows for directed links (util then holds the upward ones).
    tier_mode: util rows are per-tier congestion c[4] and a pair's bandwidth is
    B_tau (1 - c_tau) (the paper's four maps)."""
    pre = [i for i in range(tree.n) if role[i] == 0]
    dec_inst = [i for i in range(tree.n) if role[i] == 1]
    D = len(dec_inst)
    load = [0] * D
    R = len(length)
    dec = [-1] * R
    best = [None] * R
    wn, wp, wl = (frac(x) for x in w)
    th = frac(theta)
    for code in events:
        code = int(code)
        r = code & 0x7FFFFFFF
        l = int(length[r])
        if code >> 31:
            if dec[r] >= 0:
                load[dec[r]] -= l
            continue
        p = pre[int(prefill[r])]
        u_row = util[int(snap[r])]
        scores = []
        for d in range(D):
            if load[d] + l > cap:
                scores.append(None)
                continue
            miss_tok = l - 16 * int(M[r][d])
            if tier_mode:
                tau = tree.tier(p, dec_inst[d])
                b = frac(bw[tau]) * (1 - frac(u_row[tau]))
            elif util_down is None:
                b = bottleneck(tree, bw, u_row, p, dec_inst[d])
            else:
                b = bottleneck_directed(tree, bw, u_row, util_down[int(snap[r])], p, dec_inst[d])
            T = Fraction(miss_tok * bpt) / b + frac(lat[tree.tier(p, dec_inst[d])])
            scores.append(wn * T + wp * Fraction(miss_tok, l) + wl * th * load[d])
        cands = [(s, d) for d, s in enumerate(scores) if s is not None]
        if cands:
            s, d = min(cands)
            dec[r] = d
            best[r] = s
            load[d] += l
    return dec, best, load


def greedy_exact_inflight(tree, role, bw, lat, util, length, prefill, snap, arrival_us, M,
                          events, w, theta, cap, bpt, inflight_cap):
    """Exact-rational Algorithm 1 with self-contention: the effective bandwidth of a
    candidate is its path bottleneck over 1 + n[prefill][tier]; a dispatch raises that
    counter (at most inflight_cap) and its transfer completes, lowering it again (not
    below zero), at arrival + round-half-up(transfer time in microseconds); completions
    due at or before an arrival come first.  Returns (dec, best, load, xfer_us)."""
    pre = [i for i in range(tree.n) if role[i] == 0]
    dec_inst = [i for i in range(tree.n) if role[i] == 1]
    D = len(dec_inst)
    load = [0] * D
    R = len(length)
    dec = [-1] * R
    best = [None] * R
    xfer_us = [-1] * R
    n = {}                       # (prefill rank, tier) -> counter
    pending = []                 # (done time, prefill rank, tier)
    wn, wp, wl = (frac(x) for x in w)
    th = frac(theta)
    for code in events:
        code = int(code)
        r = code & 0x7FFFFFFF
        l = int(length[r])
        if code >> 31:
            if dec[r] >= 0:
                load[dec[r]] -= l
            continue
        now = int(arrival_us[r])
        pending.sort()
        while pending and pending[0][0] <= now:
            _, pr, tau = pending.pop(0)
            n[(pr, tau)] = max(0, n.get((pr, tau), 0) - 1)
        pr = int(prefill[r])
        p = pre[pr]
        u_row = util[int(snap[r])]
        scores, times = [], []
        for d in range(D):
            tau = tree.tier(p, dec_inst[d])
            miss_tok = l - 16 * int(M[r][d])
            b_eff = bottleneck(tree, bw, u_row, p, dec_inst[d]) / (1 + n.get((pr, tau), 0))
            T = Fraction(miss_tok * bpt) / b_eff + frac(lat[tau])
            times.append((T, tau))
            if load[d] + l > cap:
                scores.append(None)
                continue
            scores.append(wn * T + wp * Fraction(miss_tok, l) + wl * th * load[d])
        cands = [(s, d) for d, s in enumerate(scores) if s is not None]
        if not cands:
            continue
        s, d = min(cands)
        dec[r] = d
        best[r] = s
        load[d] += l
        T, tau = times[d]
        dt = int((T * 1000000 + Fraction(1, 2)) // 1)
        xfer_us[r] = dt
        n[(pr, tau)] = min(inflight_cap, n.get((pr, tau), 0) + 1)
        pending.append((now + dt, pr, tau))
    return dec, best, load, xfer_us


def greedy_exact_load(tree, role, bw, lat, util, length, prefill, snap, M, events, w, bpt,
                      t_a, t_b, beta_max, m_min, m0):
    """Exact-rational Algorithm 1 with the paper's compute-load model: each decode holds n
    requests and m free bytes; beta = min(n, beta_max), q = n - beta,
    T_queue = max(0, q - (beta_max - beta)) (a + b beta), T_decode = a + b (beta + 1);
    feasible iff m >= s_eff + m_min; dispatch n += 1, m -= s_eff, departure undoes it.
    Returns (dec, best, n, m)."""
    pre = [i for i in range(tree.n) if role[i] == 0]
    dec_inst = [i for i in range(tree.n) if role[i] == 1]
    D = len(dec_inst)
    n, m = [0] * D, [m0] * D
    R = len(length)
    dec, best = [-1] * R, [None] * R
    wn, wp, wl = (frac(x) for x in w)
    a, b = frac(t_a), frac(t_b)
    for code in events:
        code = int(code)
        r = code & 0x7FFFFFFF
        l = int(length[r])
        if code >> 31:
            if dec[r] >= 0:
                d = dec[r]
                n[d] -= 1
                m[d] += (l - 16 * int(M[r][d])) * bpt
            continue
        p = pre[int(prefill[r])]
        u_row = util[int(snap[r])]
        cands = []
        for d in range(D):
            miss_tok = l - 16 * int(M[r][d])
            s_eff = miss_tok * bpt
            if m[d] < s_eff + m_min:
                continue
            T = Fraction(s_eff) / bottleneck(tree, bw, u_row, p, dec_inst[d]) \
                + frac(lat[tree.tier(p, dec_inst[d])])
            beta = min(n[d], beta_max)
            q = n[d] - beta
            t_queue = max(0, q - (beta_max - beta)) * (a + b * beta)
            t_decode = a + b * (beta + 1)
            cands.append((wn * T + wp * Fraction(miss_tok, l) + wl * (t_queue + t_decode), d))
        if cands:
            s, d = min(cands)
            dec[r], best[r] = d, s
            n[d] += 1
            m[d] -= (l - 16 * int(M[r][d])) * bpt
    return dec, best, n, m


def lru_front(blocks, cache, cap):
    """A recency list (most recent first) after `blocks` are used: the distinct blocks in
    order of first appearance go to the front, the rest of the list keeps its order, and
    the list is cut to its `cap` most recent entries."""
    front = list(dict.fromkeys(int(b) for b in blocks))
    seen = set(front)
    merged = front + [k for k in cache if k not in seen]
    return merged if cap is None else merged[:cap]


def greedy_exact_evolving(tree, role, bw, lat, util, length, prefill, snap, keys_per_decode,
                          chains, events, w, theta, cap, bpt, cap_blocks=None):
    """Exact-rational Algorithm 1 with evolving caches: hits per arrival against the caches
    of that moment (a list scan to the first miss), and a dispatch brings the request's
    whole chain to the front of its decode's recency list, which keeps at most cap_blocks
    entries (None: no limit).  Returns (dec, best, load, M, caches), caches most recent
    first."""
    pre = [i for i in range(tree.n) if role[i] == 0]
    dec_inst = [i for i in range(tree.n) if role[i] == 1]
    D = len(dec_inst)
    caches = [lru_front(keys_per_decode[d], [], cap_blocks) for d in range(D)]
    load = [0] * D
    R = len(length)
    dec, best = [-1] * R, [None] * R
    M = [[0] * D for _ in range(R)]
    wn, wp, wl = (frac(x) for x in w)
    th = frac(theta)
    for code in events:
        code = int(code)
        r = code & 0x7FFFFFFF
        l = int(length[r])
        if code >> 31:
            if dec[r] >= 0:
                load[dec[r]] -= l
            continue
        chain = [int(x) for x in chains[r]]
        for d in range(D):
            M[r][d] = lcp_blocks(chain, set(caches[d]))
        p = pre[int(prefill[r])]
        u_row = util[int(snap[r])]
        cands = []
        for d in range(D):
            if load[d] + l > cap:
                continue
            miss_tok = l - 16 * M[r][d]
            T = Fraction(miss_tok * bpt) / bottleneck(tree, bw, u_row, p, dec_inst[d]) \
                + frac(lat[tree.tier(p, dec_inst[d])])
            cands.append((wn * T + wp * Fraction(miss_tok, l) + wl * th * load[d], d))
        if cands:
            s, d = min(cands)
            dec[r], best[r] = d, s
            load[d] += l
            caches[d] = lru_front(chain, caches[d], cap_blocks)
    return dec, best, load, M, caches
