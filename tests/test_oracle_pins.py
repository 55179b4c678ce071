"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test would fail on a plausible slip in the oracle: a dropped latency term,
(1 + u) for (1 - u), a swapped prefill/decode index, a transposed [s][p][d]
layout, a wrong tier, a prefix scan that skips holes, a wrong tie-break or a
load update applied at the wrong time.
"""
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
import synth
from tests import naive

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def golden(name):
    vals = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            k, v = line.split()
            vals[k] = float(v)
    return vals


# --------------------------------------------------------------------- P1: Eq. 1
def test_kv_closed_form():
    g = golden("kv_closed_form.txt")
    bpt = oracle.kv_bytes_per_token(80, 8, 128, 2)
    assert bpt == g["bytes_per_token"]
    assert bpt / 4 == g["bytes_per_token_shard_tp4"]
    s = bpt * g["context_tokens"]
    assert s == g["bytes_context"] == 5 * 2 ** 33          # exactly 40 GiB
    assert s / 4 == g["bytes_context_per_pair_tp4"] == 10 * 2 ** 30
    # 10 GB (decimal) over 25 Gbps
    t = oracle.transfer_time(g["pair_transfer_bytes_decimal"], g["link_gbps"] * 1e9 / 8, 0.0)
    assert t == pytest.approx(g["pair_transfer_seconds"], rel=1e-15)
    # the generator's per-shard constant agrees with the oracle's closed form
    assert synth.BYTES_PER_TOKEN_SHARD == bpt / 4


# --------------------------------------------------------------------- P2: worked example
def test_worked_example_formulas():
    g = golden("worked_example.txt")
    # Eq. 2
    assert oracle.s_eff(g["s_r"], g["d1_hit"] * 32768, 32768) == pytest.approx(g["s_eff_d1"], rel=1e-15)
    assert oracle.s_eff(g["s_r"], g["d2_hit"] * 32768, 32768) == pytest.approx(g["s_eff_d2"], rel=1e-12)
    # Eq. 4 with self-contention
    b1 = oracle.beff_tier(g["B2"], g["c"], g["d1_inflight"])
    b2 = oracle.beff_tier(g["B3"], g["c"], g["d2_inflight"])
    assert b1 == pytest.approx(g["beff_d1"], rel=1e-15)
    assert b2 == pytest.approx(g["beff_d2"], rel=1e-15)
    # Eq. 3
    assert oracle.transfer_time(g["s_eff_d1"], b1, 0.0) == pytest.approx(g["T_d1"], rel=1e-15)
    assert oracle.transfer_time(g["s_eff_d2"], b2, 0.0) == pytest.approx(g["T_d2"], rel=1e-15)
    b2p = oracle.beff_tier(g["B3"], g["c3_perturbed"], 0)
    assert b2p == pytest.approx(g["beff_d2_perturbed"], rel=1e-15)
    assert oracle.transfer_time(g["s_eff_d2"], b2p, 0.0) == pytest.approx(g["T_d2_perturbed"], rel=1e-15)


def test_worked_example_through_cost_matrix():
    """The per-link oracle reproduces the example's cross-pod numbers when every link
    on the path carries the tier congestion and the top-level link is the slowest."""
    g = golden("worked_example.txt")
    fanout = (1, 2, 2, 2)                 # 8 instances, two pods
    role = np.array([0, 1, 1, 1, 1, 1, 1, 1], np.uint8)   # instance 0 prefills
    bw = [4 * g["B2"], 2 * g["B2"], g["B2"], g["B3"]]
    lat = [0.0, 0.0, 0.0, 0.0]
    L = oracle.used_links(fanout)
    for c3, T_expect in ((g["c"], g["T_d2"]), (g["c3_perturbed"], g["T_d2_perturbed"])):
        u = np.full((1, L), np.float32(g["c"]), np.float32)
        # pod-spine links (level 3) get c3
        u[0, L - 2:] = np.float32(c3)
        C = oracle.cost_matrix(fanout, role, bw, lat, u, g["s_eff_d2"])
        # decode ranks 3..6 are instances 4..7: the other pod (tier 3)
        t = C[0, 0, 3]
        # fp32 utilisations: 0.2 and 0.5 are not exact in binary, so compare loosely
        assert t == pytest.approx(T_expect, rel=1e-7)
        # same-pod candidates see B2 * (1 - c) with c = 0.2 on the 1 GB payload
        assert C[0, 0, 2] == pytest.approx(g["s_eff_d2"] / (g["B2"] * 0.8), rel=1e-7)


def test_single_uncontended_path_is_top_link_plus_latency():
    """Analogue of the simulator validation statement (Sec. VI-B): an idle path moves
    data at the bandwidth of its slowest (top) link, plus the tier latency."""
    fanout = (2, 2, 2, 2)
    role = synth.roles(synth.tiny_spec())
    bw = [900e9, 400e9, 200e9, 100e9]
    lat = [1e-6, 3e-6, 6e-6, 10e-6]
    L = oracle.used_links(fanout)
    C = oracle.cost_matrix(fanout, role, bw, lat, np.zeros((1, L), np.float32), 1e9)
    pre = np.flatnonzero(role == 0)
    dec = np.flatnonzero(role == 1)
    tree = naive.ExplicitTree(fanout)
    for a, p in enumerate(pre):
        for b, d in enumerate(dec):
            tau = tree.tier(p, d)
            assert C[0, a, b] == 1e9 / bw[tau] + lat[tau]


# --------------------------------------------------------------------- topology
def test_tier_and_paths_match_explicit_graph():
    for fanout in [(2, 2, 2, 2), (1, 2, 2, 4), (3, 1, 2, 2), (1, 8, 8, 2)]:
        tree = naive.ExplicitTree(fanout)
        assert oracle.used_links(fanout) == tree.n_edges
        rng = np.random.default_rng(1)
        pairs = [(i, j) for i in range(tree.n) for j in range(tree.n)] if tree.n <= 16 else \
            [tuple(x) for x in rng.integers(0, tree.n, size=(300, 2))]
        for i, j in pairs:
            if i == j:
                continue
            links, levels = oracle.path_links(fanout, i, j)
            assert sorted(int(x) for x in links) == sorted(tree.path(i, j))
            assert oracle.tier(fanout, i, j) == tree.tier(i, j)
            # closed form of the tier from tree coordinates
            f0, f1, f2, _ = fanout
            closed = 0 if i // f0 == j // f0 else 1 if i // (f0 * f1) == j // (f0 * f1) else \
                2 if i // (f0 * f1 * f2) == j // (f0 * f1 * f2) else 3
            assert oracle.tier(fanout, i, j) == closed


# --------------------------------------------------------------------- P3: per-link oracle
def _level_util(fanout, c):
    tree = naive.ExplicitTree(fanout)
    u = np.zeros((1, tree.n_edges), np.float32)
    for e, lvl in tree.level.items():
        u[0, e] = c[lvl]
    return u


def test_per_tier_reduction_of_eq4():
    """Every link of level k at utilisation c_k: with a constant c and B0>B1>B2>B3 the
    bottleneck is B_tau (1 - c) (Eq. 4 with n_inflight = 0); in general it is
    min_{j <= tau} B_j (1 - c_j)."""
    fanout = (2, 2, 2, 2)
    role = synth.roles(synth.tiny_spec())
    bw = [900e9, 400e9, 200e9, 100e9]
    lat = [1e-6, 3e-6, 6e-6, 10e-6]
    tree = naive.ExplicitTree(fanout)
    pre = np.flatnonzero(role == 0)
    dec = np.flatnonzero(role == 1)
    kv = 7.5e9
    for c in ([0.25] * 4, [0.0, 0.5, 0.75, 0.125], [0.875, 0.0, 0.5, 0.0]):
        u = _level_util(fanout, c)
        C = oracle.cost_matrix(fanout, role, bw, lat, u, kv)
        for a, p in enumerate(pre):
            for b, d in enumerate(dec):
                tau = tree.tier(p, d)
                bb = min(bw[j] * (1 - c[j]) for j in range(tau + 1))
                assert C[0, a, b] == pytest.approx(kv / bb + lat[tau], rel=1e-15)
                if len(set(c)) == 1:
                    assert C[0, a, b] == pytest.approx(kv / (bw[tau] * (1 - c[0])) + lat[tau], rel=1e-15)


def test_cost_matrix_random_links_exact_vs_bfs():
    """Random per-link utilisations, P != D (catches a transposed layout or swapped
    endpoints): the oracle equals the exact-rational BFS evaluation."""
    fanout = (2, 2, 2, 2)
    tree = naive.ExplicitTree(fanout)
    role = (np.arange(tree.n) % 3 != 0).astype(np.uint8)     # P = 6, D = 10
    bw = [900e9, 400e9, 200e9, 100e9]
    lat = [1e-6, 3e-6, 6e-6, 10e-6]
    rng = np.random.default_rng(7)
    u = rng.uniform(0, 0.95, size=(3, tree.n_edges + 5)).astype(np.float32)   # padded links
    kv = 3.3e9
    C = oracle.cost_matrix(fanout, role, bw, lat, u, kv)
    pre = np.flatnonzero(role == 0)
    dec = np.flatnonzero(role == 1)
    assert C.shape == (3, len(pre), len(dec))
    for s in range(3):
        for a, p in enumerate(pre):
            for b, d in enumerate(dec):
                exact = naive.cost(tree, bw, lat, u[s], p, d, kv)
                assert Fraction(C[s, a, b]) == pytest.approx(exact, rel=1e-15)
    # sampled entries agree with the full matrix
    s = rng.integers(0, 3, 50); a = rng.integers(0, len(pre), 50); b = rng.integers(0, len(dec), 50)
    e = oracle.cost_entries(fanout, role, bw, lat, u, s, a, b, kv)
    np.testing.assert_array_equal(e, C[s, a, b])


def test_up_bottleneck_consistent_with_paths():
    fanout = (2, 2, 2, 2)
    tree = naive.ExplicitTree(fanout)
    bw = [900e9, 400e9, 200e9, 100e9]
    rng = np.random.default_rng(3)
    u = rng.uniform(0, 0.9, size=(2, tree.n_edges)).astype(np.float32)
    UB = oracle.up_bottleneck(fanout, bw, u)
    for s in range(2):
        for i in range(tree.n):
            for j in range(tree.n):
                if i == j:
                    continue
                tau = tree.tier(i, j)
                bb = naive.bottleneck(tree, bw, u[s], i, j)
                assert min(UB[s, i, tau], UB[s, j, tau]) == pytest.approx(float(bb), rel=1e-15)
            # monotone non-increasing in k
            assert all(UB[s, i, k + 1] <= UB[s, i, k] for k in range(3))


# --------------------------------------------------------------------- P7: prefix LCP
def test_prefix_first_miss_semantics():
    chain = np.array([11, 22, 33, 44], np.uint64)
    off = np.array([0, 4], np.uint64)
    for cache, m in (([11, 33, 44], 1), ([22, 33, 44], 0), ([11, 22, 33, 44, 99], 4),
                     ([44, 33, 22, 11], 4), ([], 0), ([11, 22, 44], 2)):
        got = oracle.prefix_match_one(np.array(cache, np.uint64), chain, off)
        assert int(got[0]) == m == naive.lcp_blocks(list(chain), cache)
    # an empty chain matches zero blocks
    got = oracle.prefix_match_one(np.array([1, 2], np.uint64), np.zeros(0, np.uint64),
                                  np.array([0, 0], np.uint64))
    assert int(got[0]) == 0


def test_prefix_closed_form_under_generator():
    """Chains are a root prefix followed by a never-cached tail and caches hold root
    prefixes of depth delta: M = min(shared_r, delta_{d, root_r})."""
    spec = synth.tiny_spec()
    w = synth.make_workload(spec)
    keys = [w.keys(g, d) for g in range(w.n_sets) for d in range(w.D)]
    key_off = np.concatenate([[0], np.cumsum([len(k) for k in keys])]).astype(np.uint64)
    M = oracle.prefix_match(np.concatenate(keys), key_off, w.D, w.chains(), w.chain_off, w.set_off)
    set_of = synth.request_set(w)
    expect = np.minimum(w.shared[:, None].astype(np.int64),
                        w.depth[set_of, :, :][np.arange(w.R), :, w.root.astype(np.int64)])
    np.testing.assert_array_equal(M.astype(np.int64), expect)
    # the generator's own statement of it, used where the oracle's sets do not fit
    np.testing.assert_array_equal(synth.constructed_hits(w), M)
    np.testing.assert_array_equal(synth.constructed_hits(w, 7, 29), M[7:29])
    assert (M > 0).any() and (M.astype(np.int64) < (w.chain_off[1:] - w.chain_off[:-1])[:, None]).any()


# --------------------------------------------------------------------- P4: greedy
def _tiny_problem(seed, D_role="alternate", R=6, cap=None, n_snap=3, span=1000):
    rng = np.random.default_rng(seed)
    fanout = (2, 2, 2, 1) if D_role == "alternate" else (2, 2, 2, 2)
    tree = naive.ExplicitTree(fanout)
    role = (np.arange(tree.n) % 2).astype(np.uint8)       # P = D = 4
    bw = [900e9, 400e9, 200e9, 100e9]
    lat = [1e-6, 3e-6, 6e-6, 10e-6]
    u = rng.uniform(0, 0.9, size=(n_snap, tree.n_edges)).astype(np.float32)
    D = int(role.sum()); P = tree.n - D
    length = rng.integers(16, 4000, size=R).astype(np.uint32)
    prefill = rng.integers(0, P, size=R).astype(np.uint32)
    snap = rng.integers(0, n_snap, size=R).astype(np.uint32)
    M = np.zeros((R, D), np.uint16)
    for r in range(R):
        M[r] = rng.integers(0, int(length[r]) // 16 + 1, size=D)
    # events: arrivals in order, departures interleaved after their arrival
    t_arr = np.sort(rng.integers(0, span, size=R))
    t_dep = t_arr + rng.integers(1, 600 * span // 1000, size=R)
    t = np.concatenate([t_dep, t_arr]); typ = np.concatenate([np.zeros(R), np.ones(R)]).astype(int)
    rr = np.concatenate([np.arange(R), np.arange(R)])
    o = np.lexsort((rr, typ, t))
    events = (rr[o].astype(np.uint64) | ((1 - typ[o]).astype(np.uint64) << np.uint64(31))).astype(np.uint32)
    cap = int(cap if cap is not None else rng.integers(3000, 9000))
    return dict(tree=tree, fanout=fanout, role=role, bw=bw, lat=lat, u=u, length=length,
                prefill=prefill, snap=snap, M=M, events=events, cap=cap, arrival_us=t_arr)


def _run_oracle(pb, w, theta=float(np.float32(1e-6)), bpt=81920, hint=None):
    return oracle.schedule_stream(pb["fanout"], pb["role"], pb["bw"], pb["lat"], pb["u"],
                                  pb["length"], pb["prefill"], pb["snap"], pb["M"], pb["events"],
                                  w[0], w[1], w[2], theta, pb["cap"], bpt, hint=hint)


def test_greedy_matches_exact_rational_bruteforce():
    theta = float(np.float32(1e-6))
    n_cmp = 0
    for seed in range(40):
        pb = _tiny_problem(seed)
        w = tuple(float(np.float32(x)) for x in np.random.default_rng(100 + seed).uniform(0, 2, 3))
        res = _run_oracle(pb, w)
        dec, best, load = naive.greedy_exact(pb["tree"], pb["role"], pb["bw"], pb["lat"], pb["u"],
                                             pb["length"], pb["prefill"], pb["snap"], pb["M"],
                                             pb["events"], w, theta, pb["cap"], 81920)
        assert list(res.dec) == dec
        for r in range(len(dec)):
            if dec[r] >= 0:
                assert res.best[r] == pytest.approx(float(best[r]), rel=1e-14)
                n_cmp += 1
            else:
                assert np.isinf(res.best[r])
        assert list(res.load) == load
    assert n_cmp > 100


def test_greedy_rejects_when_nothing_feasible():
    pb = _tiny_problem(5, cap=20)                 # every request is longer than the capacity
    res = _run_oracle(pb, (1.0, 1.0, 1.0))
    assert (res.dec == -1).all() and res.rejects == len(res.dec)
    assert np.isinf(res.best).all() and np.isinf(res.second).all()
    assert (res.load == 0).all()


def _independent_cache_load(pb, wp, wl, theta):
    """Cache + load scorer written without any network term (the CLA-style reduction)."""
    D = int(pb["role"].sum())
    load = [0] * D
    R = len(pb["length"])
    dec = [-1] * R
    for code in pb["events"]:
        code = int(code); r = code & 0x7FFFFFFF; l = int(pb["length"][r])
        if code >> 31:
            if dec[r] >= 0:
                load[dec[r]] -= l
            continue
        best = None
        for d in range(D):
            if load[d] + l > pb["cap"]:
                continue
            s = Fraction(wp) * Fraction(l - 16 * int(pb["M"][r][d]), l) + Fraction(wl) * Fraction(theta) * load[d]
            if best is None or s < best[0]:
                best = (s, d)
        if best is not None:
            dec[r] = best[1]
            load[best[1]] += l
    return dec


def test_greedy_reductions():
    theta = float(np.float32(1e-6))
    for seed in range(25):
        pb = _tiny_problem(seed)
        # (ii) network weight zero: a cache + load scorer
        res = _run_oracle(pb, (0.0, 1.0, 1.0))
        assert list(res.dec) == _independent_cache_load(pb, 1.0, 1.0, theta)
        # (iii) only load: least loaded feasible, lowest index among equals
        res = _run_oracle(pb, (0.0, 0.0, 1.0))
        assert list(res.dec) == _independent_cache_load(pb, 0.0, 1.0, theta)
        # (iv) all weights zero: the lowest feasible index
        res = _run_oracle(pb, (0.0, 0.0, 0.0))
        assert list(res.dec) == _independent_cache_load(pb, 0.0, 0.0, theta)


def test_greedy_lowest_index_tie_break_and_second():
    pb = _tiny_problem(11, cap=10 ** 9)
    pb["M"][:] = 0
    res = _run_oracle(pb, (0.0, 1.0, 0.0))        # every candidate has miss = 1: all tie
    arrivals = [int(c) & 0x7FFFFFFF for c in pb["events"] if not (int(c) >> 31)]
    for r in arrivals:
        assert res.dec[r] == 0
        assert res.best[r] == res.second[r] == 1.0


def test_greedy_load_accounting_on_truncated_events():
    """Loads after a prefix of the events equal the tokens of dispatched requests whose
    departure has not been processed yet."""
    pb = _tiny_problem(21, R=6, cap=10 ** 9)
    full = pb["events"]
    for cut in range(1, len(full) + 1):
        pb["events"] = full[:cut]
        res = _run_oracle(pb, (1.0, 1.0, 1.0))
        D = int(pb["role"].sum())
        expect = np.zeros(D, np.int64)
        for code in full[:cut]:
            code = int(code); r = code & 0x7FFFFFFF
            sign = -1 if code >> 31 else 1
            expect[res.dec[r]] += sign * int(pb["length"][r])
        np.testing.assert_array_equal(res.load, expect)
    assert (res.load == 0).all()                  # every request departed by the end


def test_hint_replay_counts():
    pb = _tiny_problem(2, cap=10 ** 9)
    w = (1.0, 1.0, 1.0)
    ref = _run_oracle(pb, w)
    same = _run_oracle(pb, w, hint=ref.dec.copy())
    assert same.near_ties == 0 and same.mismatches == 0
    np.testing.assert_array_equal(same.dec, ref.dec)
    # a hint that differs away from a tie is a mismatch and is adopted
    arrivals = [int(c) & 0x7FFFFFFF for c in pb["events"] if not (int(c) >> 31)]
    h = ref.dec.copy()
    r0 = arrivals[0]
    h[r0] = (h[r0] + 1) % int(pb["role"].sum())
    got = _run_oracle(pb, w, hint=h)
    assert got.mismatches >= 1 and got.dec[r0] == h[r0]
    # exact ties: any index among the tied minimum is accepted as a near-tie
    pb["M"][:] = 0
    tie = _run_oracle(pb, (0.0, 1.0, 0.0), hint=np.full(len(pb["length"]), 2, np.int32))
    assert tie.mismatches == 0 and tie.near_ties == len(arrivals)


# --------------------------------------------------------------------- P5: Proposition 1
def _prop1_problem(ell, rho2, c=0.3):
    fanout = (1, 2, 2, 2)            # 8 instances: nodes = instances; leaves of 2; pods of 2 leaves
    # instance 0 prefills; instance 1 (same leaf: tier 1) and instance 4 (other pod: tier 3) decode
    role = np.array([0, 1, 0, 0, 1, 0, 0, 0], np.uint8)
    B1 = 100e9 / 8
    bw = [4 * B1, B1, B1 / 2, B1 / 4]      # k = B1 / B3 = 4
    L = oracle.used_links(fanout)
    u = np.full((1, L), np.float32(c), np.float32)
    M = np.array([[0, int(rho2 * ell) // 16]], np.uint16)   # d1 cold, d2 warm
    return dict(fanout=fanout, role=role, bw=bw, lat=[0.0] * 4, u=u,
                length=np.array([ell], np.uint32), prefill=np.zeros(1, np.uint32),
                snap=np.zeros(1, np.uint32), M=M,
                events=np.array([0, 1 << 31], np.uint32), cap=10 ** 9)


def test_proposition1_family():
    g = golden("propositions.txt")
    gaps = []
    for ell in [2 ** k for k in range(10, 18)]:
        pb = _prop1_problem(ell, g["prop1_rho2"])
        cache_only = _run_oracle(pb, (0.0, 1.0, 0.0))
        net = _run_oracle(pb, (1.0, 0.0, 0.0))
        assert cache_only.dec[0] == 1          # the warm cross-pod instance
        assert net.dec[0] == 0                 # the cold same-leaf instance
        t_d1, t_d2 = net.best[0], net.second[0]
        assert t_d2 / t_d1 == pytest.approx(g["prop1_transfer_ratio"], rel=1e-6)
        gaps.append(t_d2 - t_d1)
    # the additive gap grows linearly with context length: arbitrarily worse
    for a, b in zip(gaps, gaps[1:]):
        assert b / a == pytest.approx(2.0, rel=1e-6)
    assert g["prop1_lhs"] < g["prop1_k"] * (1 - g["prop1_rho2"]) == g["prop1_rhs"]


def test_proposition1_inequality_matches_oracle_choice():
    rng = np.random.default_rng(0)
    checked = 0
    for _ in range(400):
        ell = int(rng.integers(1024, 65536))
        rho1, rho2 = sorted(rng.uniform(0, 0.95, 2))
        c1, c3 = rng.uniform(0, 0.9, 2)
        pb = _prop1_problem(ell, 0.0)
        n = ell // 16
        m1, m2 = int(rho1 * n), int(rho2 * n)
        pb["M"] = np.array([[m1, m2]], np.uint16)
        L = pb["u"].shape[1]
        tree = naive.ExplicitTree(pb["fanout"])
        for e, lvl in tree.level.items():
            pb["u"][0, e] = np.float32(c1 if lvl <= 1 else c3)
        B1, B3 = pb["bw"][1], pb["bw"][3]
        c1f, c3f = float(pb["u"][0, 0]), float(pb["u"][0, L - 1])
        if B3 * (1 - c3f) > pb["bw"][1] * (1 - c1f):
            continue                      # the proposition's tier-3 bottleneck must be the top link
        r1 = 16 * m1 / ell; r2 = 16 * m2 / ell
        k = B1 / B3
        lhs, rhs = (1 - r1), k * (1 - c1f) / (1 - c3f) * (1 - r2)
        if abs(lhs - rhs) < 1e-9 * max(lhs, rhs):
            continue
        net = _run_oracle(pb, (1.0, 0.0, 0.0))
        assert (net.dec[0] == 0) == (lhs < rhs)
        checked += 1
    assert checked > 100


# --------------------------------------------------------------------- P6: Proposition 2
def test_proposition2_numeric_bound():
    g = golden("propositions.txt")
    k, c = g["prop2_ratio"], g["prop2_c"]
    bound = (k * (1 - c) - 1 * (1 - c)) / (k + 1)
    assert bound == pytest.approx(g["prop2_bound"], rel=1e-12)


def test_proposition2_ranking_robustness():
    """Tier ranking of the oracle's transfer cost survives any stale perturbation below
    the bound and is inverted by the worst case just above it."""
    fanout = (1, 2, 2, 2)
    role = np.array([0, 1, 0, 0, 1, 0, 0, 0], np.uint8)     # d at tier 1 and tier 3
    tree = naive.ExplicitTree(fanout)
    rng = np.random.default_rng(9)
    tested = 0
    for _ in range(300):
        Bt = float(rng.uniform(20e9, 100e9)); Btp = float(rng.uniform(2e9, Bt))
        ct, ctp = rng.uniform(0, 0.9, 2)
        if Bt * (1 - ct) <= Btp * (1 - ctp):
            continue
        eps = (Bt * (1 - ct) - Btp * (1 - ctp)) / (Bt + Btp)
        bw = [1e15, Bt, 1e15, Btp]       # only the tier-1 and tier-3 links can bind
        def order(c_t, c_tp):
            u = np.zeros((1, tree.n_edges), np.float32)
            for e, lvl in tree.level.items():
                u[0, e] = np.float32(c_t if lvl <= 1 else c_tp)
            C = oracle.cost_matrix(fanout, role, bw, [0.0] * 4, u, 1e9)
            return C[0, 0, 0] < C[0, 0, 1]       # the faster tier costs less
        assert order(ct, ctp)
        for _ in range(5):
            d1, d2 = rng.uniform(-0.98 * eps, 0.98 * eps, 2)
            a, b = ct + d1, ctp + d2
            if 0 <= a < 1 and 0 <= b < 1 and eps > 1e-3:
                assert order(a, b)
        a, b = ct + 1.05 * eps, ctp - 1.05 * eps
        if eps > 1e-3 and 0 <= a < 1 and 0 <= b < 1:
            assert not order(a, b)
            tested += 1
    assert tested > 30


def test_prefix_match_tables_with_holes():
    """Multi-table form: two sets of two caches each, caches with holes in the chain."""
    chains = np.array([1, 2, 3, 4, 5,   1, 2, 3,   9, 2, 3], np.uint64)
    chain_off = np.array([0, 5, 8, 11], np.uint64)
    set_off = np.array([0, 2, 3], np.uint32)           # set 0: requests 0,1; set 1: request 2
    caches = [[1, 2, 4, 5], [1, 2, 3, 4, 5],           # set 0, decodes 0 and 1
              [2, 3, 9], [9, 3]]                       # set 1, decodes 0 and 1
    keys = np.concatenate([np.array(c, np.uint64) for c in caches])
    key_off = np.concatenate([[0], np.cumsum([len(c) for c in caches])]).astype(np.uint64)
    M = oracle.prefix_match(keys, key_off, 2, chains, chain_off, set_off)
    expect = [[2, 5], [2, 3], [3, 1]]
    np.testing.assert_array_equal(M, np.array(expect, np.uint16))
    for r in range(3):
        g = 0 if r < 2 else 1
        for d in range(2):
            assert M[r, d] == naive.lcp_blocks(list(chains[chain_off[r]:chain_off[r + 1]]),
                                               caches[2 * g + d])


def test_greedy_capacity_boundary_is_inclusive():
    """Line 1 of Algorithm 1 keeps a candidate whose free capacity equals the demand."""
    pb = _tiny_problem(4, R=6)
    l0 = int(pb["length"][0])
    pb["cap"] = l0
    res = _run_oracle(pb, (1.0, 1.0, 1.0))
    assert res.dec[0] >= 0
    pb["cap"] = l0 - 1
    res = _run_oracle(pb, (1.0, 1.0, 1.0))
    assert res.dec[0] == -1


# ------------------------------------------------ self-contention (NEXT: n_inflight)
def _run_inflight(pb, w, inflight_cap, theta=float(np.float32(1e-6)), bpt=81920):
    return oracle.schedule_stream_inflight(pb["fanout"], pb["role"], pb["bw"], pb["lat"], pb["u"],
                                           pb["length"], pb["prefill"], pb["snap"],
                                           pb["arrival_us"], pb["M"], pb["events"], w[0], w[1],
                                           w[2], theta, pb["cap"], bpt, inflight_cap)


def test_inflight_off_is_the_plain_greedy():
    """A cap of 0 keeps every counter at 0: the plain Algorithm 1, value for value."""
    for seed in range(20):
        pb = _tiny_problem(seed, span=50_000)
        w = tuple(float(np.float32(x)) for x in np.random.default_rng(300 + seed).uniform(0, 2, 3))
        a, b = _run_oracle(pb, w), _run_inflight(pb, w, 0)
        np.testing.assert_array_equal(a.dec, b.dec)
        np.testing.assert_array_equal(a.best, b.best)
        np.testing.assert_array_equal(a.second, b.second)
        np.testing.assert_array_equal(a.load, b.load)
        assert ((b.xfer_us >= 0) == (b.dec >= 0)).all()


def test_inflight_matches_exact_rational_bruteforce():
    """Counters, completions and transfer times against an exact-rational evaluator with
    BFS paths, over caps 1, 2, 3, 16 and arrivals packed into 1 ms up to spread over 0.3 s."""
    theta = float(np.float32(1e-6))
    changed = n_cmp = 0
    for seed in range(48):
        span = (1000, 50_000, 300_000)[seed % 3]
        icap = (1, 2, 3, 16)[seed % 4]
        pb = _tiny_problem(seed, R=8, span=span)
        w = tuple(float(np.float32(x)) for x in np.random.default_rng(500 + seed).uniform(0, 2, 3))
        res = _run_inflight(pb, w, icap)
        dec, best, load, xfer = naive.greedy_exact_inflight(
            pb["tree"], pb["role"], pb["bw"], pb["lat"], pb["u"], pb["length"], pb["prefill"],
            pb["snap"], pb["arrival_us"], pb["M"], pb["events"], w, theta, pb["cap"], 81920, icap)
        assert list(res.dec) == dec
        assert list(res.load) == load
        assert list(res.xfer_us) == xfer
        for r in range(len(dec)):
            if dec[r] >= 0:
                assert res.best[r] == pytest.approx(float(best[r]), rel=1e-14)
                n_cmp += 1
        plain = _run_inflight(pb, w, 0)
        changed += int((plain.dec != res.dec).any() or (plain.best != res.best).any())
    assert n_cmp > 200 and changed > 10


def _worked_example_stream(arrival_us, M_rows, c3=0.2):
    """The worked example of Sec. III-D on a (2,2,2,2) tree: prefill instance 0, decode d1 =
    instance 4 (same pod: tier 2) and d2 = instance 8 (other pod: tier 3); B2 = 6.25 GB/s,
    B3 = 3.125 GB/s (B0, B1 larger), every link at c = 0.2 except the pod-spine links of
    the path to d2 at c3; no latency.  Requests of 100,000 tokens at 100,000 B per token
    (10 GB aggregate KV), so a hit of M blocks leaves (100,000 - 16 M) * 1e5 bytes."""
    fanout = (2, 2, 2, 2)
    role = np.zeros(16, np.uint8)
    role[[4, 8]] = 1
    L = oracle.used_links(fanout)
    u = np.full((1, L), 0.2, np.float32)
    links, levels = oracle.path_links(fanout, 0, 8)
    u[0, links[levels == 3]] = c3
    R = len(arrival_us)
    t = np.asarray(arrival_us, np.int64)
    events = np.concatenate([np.arange(R), np.arange(R) | (1 << 31)]).astype(np.uint32)
    return dict(fanout=fanout, role=role, bw=[100e9, 50e9, 6.25e9, 3.125e9], lat=[0.0] * 4,
                u=u, length=np.full(R, 100_000, np.uint32), prefill=np.zeros(R, np.uint32),
                snap=np.zeros(R, np.uint32), M=np.asarray(M_rows, np.uint16), events=events,
                cap=10 ** 7, arrival_us=t)


def _worked(pb, icap):
    return oracle.schedule_stream_inflight(pb["fanout"], pb["role"], pb["bw"], pb["lat"], pb["u"],
                                           pb["length"], pb["prefill"], pb["snap"],
                                           pb["arrival_us"], pb["M"], pb["events"], 1.0, 0.0,
                                           0.0, 0.0, pb["cap"], 100_000, icap)


def test_inflight_worked_example_end_to_end():
    """Sec. III-D through the greedy: request A (no hits) goes to d1 and stays in flight
    for 2 s; request B 1 ms later (50% hit on d1, 90% on d2) sees B_eff = 2.5 GB/s on both
    candidates, T_d1 = 2.0 s and T_d2 = 0.4 s, and with c3 = 0.5, T_d2 = 0.64 s."""
    g = golden("worked_example.txt")
    a_rows = [[0, 0], [3125, 5625]]          # 3125 blocks = 50%, 5625 blocks = 90% of 6250
    res = _worked(_worked_example_stream([0, 1000], a_rows), 16)
    assert list(res.dec) == [0, 1]
    assert res.xfer_us[0] == 2_000_000                       # 10 GB at 5 GB/s
    assert res.best[1] == pytest.approx(g["T_d2"], rel=1e-6)
    assert res.second[1] == pytest.approx(g["T_d1"], rel=1e-6)   # d1 with one in flight
    assert res.xfer_us[1] == round(g["T_d2"] * 1e6)
    # the counter is what doubles d1's time: without it d1 costs 1.0 s
    off = _worked(_worked_example_stream([0, 1000], a_rows), 0)
    assert off.second[1] == pytest.approx(g["T_d1"] / 2, rel=1e-6)
    # c3 raised to 0.5 on d2's path
    pert = _worked(_worked_example_stream([0, 1000], a_rows, c3=g["c3_perturbed"]), 16)
    assert pert.best[1] == pytest.approx(g["T_d2_perturbed"], rel=1e-6)
    assert pert.second[1] == pytest.approx(g["T_d1"], rel=1e-6)


def test_inflight_completion_timing_and_cap():
    """A's transfer ends at 2,000,000 us: an arrival at that instant sees it done, one a
    microsecond earlier does not.  The counter saturates at the cap and, being a counter,
    drops on the first completion even while a second transfer is still in flight."""
    a_rows = [[0, 0], [3125, 5625]]
    at = _worked(_worked_example_stream([0, 2_000_000], a_rows), 16)
    before = _worked(_worked_example_stream([0, 1_999_999], a_rows), 16)
    assert at.second[1] == pytest.approx(1.0, rel=1e-6)
    assert before.second[1] == pytest.approx(2.0, rel=1e-6)
    # A1, A2 to d1 (the second sees one in flight: 4.0 s on d1 vs 4.0 s on d2 -> d1, the
    # lower rank), then C probes the counter: 3.0 s with the cap at 16 (two in flight),
    # 2.0 s with the cap at 1
    rows = [[0, 0], [0, 0], [3125, 5625]]
    t = [0, 10, 20]
    c16 = _worked(_worked_example_stream(t, rows), 16)
    c1 = _worked(_worked_example_stream(t, rows), 1)
    assert list(c16.dec[:2]) == [0, 0] and list(c1.dec[:2]) == [0, 0]
    assert c16.second[2] == pytest.approx(3.0, rel=1e-6)
    assert c1.second[2] == pytest.approx(2.0, rel=1e-6)
    # A1 ends at 2 s and A2 (4 s, dispatched with one in flight) at 10 us + 4 s: at
    # 2,000,005 us one completion has lowered the saturated counter to 0 although A2 is
    # still in flight
    late = _worked(_worked_example_stream([0, 10, 2_000_005], rows), 1)
    assert list(late.xfer_us[:2]) == [2_000_000, 4_000_000]
    assert late.second[2] == pytest.approx(1.0, rel=1e-6)


# ------------------------------------------------- directed links (NEXT: per direction)
def test_directed_with_equal_rows_is_undirected():
    """Equal upward and downward rows give the undirected matrix, level bottlenecks and
    greedy, value for value."""
    rng = np.random.default_rng(41)
    for fanout in ((2, 2, 2, 2), (1, 2, 3, 2)):
        tree = naive.ExplicitTree(fanout)
        role = (np.arange(tree.n) % 3 == 1).astype(np.uint8)
        bw, lat = [900e9, 400e9, 200e9, 100e9], [1e-6, 3e-6, 6e-6, 10e-6]
        u = rng.uniform(0, 0.9, size=(3, tree.n_edges)).astype(np.float32)
        np.testing.assert_array_equal(oracle.cost_matrix_directed(fanout, role, bw, lat, u, u, 1e9),
                                      oracle.cost_matrix(fanout, role, bw, lat, u, 1e9))
        np.testing.assert_array_equal(oracle.level_bottleneck_directed(fanout, role, bw, u, u),
                                      oracle.up_bottleneck(fanout, bw, u))
    for seed in range(10):
        pb = _tiny_problem(seed)
        w = (0.7, 1.1, 0.4)
        a = _run_oracle(pb, w)
        b = oracle.schedule_stream(pb["fanout"], pb["role"], pb["bw"], pb["lat"], pb["u"],
                                   pb["length"], pb["prefill"], pb["snap"], pb["M"], pb["events"],
                                   w[0], w[1], w[2], float(np.float32(1e-6)), pb["cap"], 81920,
                                   util_down=pb["u"])
        np.testing.assert_array_equal(a.dec, b.dec)
        np.testing.assert_array_equal(a.best, b.best)


def test_directed_matrix_matches_exact_rational_bfs():
    """Every (snapshot, prefill, decode) against the exact-rational evaluator that takes
    each step of the BFS path at the utilisation of its direction; P != D, all tiers."""
    rng = np.random.default_rng(42)
    for fanout, rule in (((2, 2, 2, 2), 3), ((2, 3, 2, 2), 2)):
        tree = naive.ExplicitTree(fanout)
        role = (np.arange(tree.n) % rule == 0).astype(np.uint8)
        bw, lat = [900e9, 400e9, 200e9, 100e9], [1e-6, 3e-6, 6e-6, 10e-6]
        up = rng.uniform(0, 0.95, size=(2, tree.n_edges)).astype(np.float32)
        down = rng.uniform(0, 0.95, size=(2, tree.n_edges)).astype(np.float32)
        C = oracle.cost_matrix_directed(fanout, role, bw, lat, up, down, 2.5e9)
        pre = [i for i in range(tree.n) if role[i] == 0]
        dec = [i for i in range(tree.n) if role[i] == 1]
        taus = set()
        for s in range(2):
            for a, p in enumerate(pre):
                for b, d in enumerate(dec):
                    exact = naive.frac(2.5e9) / naive.bottleneck_directed(tree, bw, up[s], down[s], p, d) \
                        + naive.frac(lat[tree.tier(p, d)])
                    assert C[s, a, b] == pytest.approx(float(exact), rel=1e-14)
                    taus.add(tree.tier(p, d))
        assert taus == {0, 1, 2, 3}
        # and the level bottlenecks the library's kernels consume
        UB = oracle.level_bottleneck_directed(fanout, role, bw, up, down)
        for s in range(2):
            for i in range(tree.n):
                row = up[s] if role[i] == 0 else down[s]
                for k in range(4):
                    climb = [naive.frac(bw[h]) * (1 - naive.frac(row[e]))
                             for h, e in enumerate(_up_links(tree, i)[:k + 1])]
                    assert UB[s, i, k] == pytest.approx(float(min(climb)), rel=1e-14)


def _up_links(tree, i):
    """Links from instance i up to the spine, level 0..3, read off the explicit tree."""
    v, out = ("inst", i), []
    height = {"inst": 0, "node": 1, "leaf": 2, "pod": 3, "spine": 4}
    while v[0] != "spine":
        for w, e in tree.adj[v]:
            if height[w[0]] == height[v[0]] + 1:
                out.append(e)
                v = w
                break
    return out


def test_directed_links_use_the_direction_crossed():
    """A congested upward level-0 link of the prefill slows every transfer from it; the
    same congestion on that link's downward direction slows none of them (the prefill
    only sends), and on a decode's downward level-0 link only the transfers to it."""
    fanout = (2, 2, 2, 2)
    role = (np.arange(16) % 2).astype(np.uint8)        # even instances prefill, odd decode
    bw, lat = [900e9, 400e9, 200e9, 100e9], [0.0] * 4
    L = oracle.used_links(fanout)
    base = np.zeros((1, L), np.float32)
    clean = oracle.cost_matrix_directed(fanout, role, bw, lat, base, base, 1e9)
    up = base.copy(); up[0, 0] = 0.99                 # instance 0's level-0 link, upward
    C = oracle.cost_matrix_directed(fanout, role, bw, lat, up, base, 1e9)
    np.testing.assert_allclose(C[0, 0], 1e9 / (900e9 * (1.0 - float(np.float32(0.99)))), rtol=1e-12)
    np.testing.assert_array_equal(C[0, 1:], clean[0, 1:])
    C = oracle.cost_matrix_directed(fanout, role, bw, lat, base, up, 1e9)
    np.testing.assert_array_equal(C, clean)           # downward on a prefill's link: unused
    down = base.copy(); down[0, 1] = 0.99             # instance 1 (decode rank 0), downward
    C = oracle.cost_matrix_directed(fanout, role, bw, lat, base, down, 1e9)
    np.testing.assert_allclose(C[0, :, 0], 1e9 / (900e9 * (1.0 - float(np.float32(0.99)))), rtol=1e-12)
    np.testing.assert_array_equal(C[0, :, 1:], clean[0, :, 1:])


def test_directed_greedy_matches_exact_rational_bruteforce():
    theta = float(np.float32(1e-6))
    for seed in range(20):
        pb = _tiny_problem(seed)
        down = np.random.default_rng(900 + seed).uniform(0, 0.9, size=pb["u"].shape).astype(np.float32)
        w = tuple(float(np.float32(x)) for x in np.random.default_rng(700 + seed).uniform(0, 2, 3))
        res = oracle.schedule_stream(pb["fanout"], pb["role"], pb["bw"], pb["lat"], pb["u"],
                                     pb["length"], pb["prefill"], pb["snap"], pb["M"], pb["events"],
                                     w[0], w[1], w[2], theta, pb["cap"], 81920, util_down=down)
        dec, best, load = naive.greedy_exact(pb["tree"], pb["role"], pb["bw"], pb["lat"], pb["u"],
                                             pb["length"], pb["prefill"], pb["snap"], pb["M"],
                                             pb["events"], w, theta, pb["cap"], 81920, util_down=down)
        assert list(res.dec) == dec and list(res.load) == load
        for r in range(len(dec)):
            if dec[r] >= 0:
                assert res.best[r] == pytest.approx(float(best[r]), rel=1e-14)


# ------------------------------------- paper-literal per-tier oracle (NEXT: four maps)
def test_per_tier_worked_example():
    """Sec. III-D with the paper's per-tier maps (no transfer in flight): d1 on tier 2 at
    B2 (1 - c) = 5 GB/s, d2 on tier 3 at 2.5 GB/s and, with c3 = 0.5, 1.5625 GB/s."""
    g = golden("worked_example.txt")
    fanout = (2, 2, 2, 2)
    role = np.zeros(16, np.uint8)
    role[[4, 8]] = 1
    bw = [100e9, 50e9, g["B2"], g["B3"]]
    c = np.full((1, 4), g["c"], np.float32)
    C5 = oracle.cost_matrix_tiers(fanout, role, bw, [0.0] * 4, c, g["s_eff_d1"])
    C1 = oracle.cost_matrix_tiers(fanout, role, bw, [0.0] * 4, c, g["s_eff_d2"])
    # d1 without the in-flight transfer: half of the example's 2.0 s
    assert C5[0, 0, 0] == pytest.approx(g["T_d1"] / 2, rel=1e-7)
    assert C1[0, 0, 1] == pytest.approx(g["T_d2"], rel=1e-7)
    c[0, 3] = g["c3_perturbed"]
    C1 = oracle.cost_matrix_tiers(fanout, role, bw, [0.0] * 4, c, g["s_eff_d2"])
    assert C1[0, 0, 1] == pytest.approx(g["T_d2_perturbed"], rel=1e-7)
    assert C1[0, 0, 0] == pytest.approx(g["s_eff_d2"] / (g["B2"] * (1 - float(np.float32(g["c"])))), rel=1e-12)


def test_per_tier_is_the_per_link_model_only_when_the_tier_level_is_the_bottleneck():
    """With every level-k link at c_k the per-link oracle takes min over levels <= tau of
    B_k (1 - c_k); the per-tier oracle takes B_tau (1 - c_tau).  They agree when that is
    the minimum and differ when a lower level is congested harder."""
    rng = np.random.default_rng(77)
    fanout = (2, 2, 2, 2)
    tree = naive.ExplicitTree(fanout)
    role = (np.arange(16) % 2).astype(np.uint8)
    bw, lat = [900e9, 400e9, 200e9, 100e9], [1e-6, 3e-6, 6e-6, 10e-6]
    level = np.array([tree.level[e] for e in range(tree.n_edges)])
    for c in ([0.1, 0.2, 0.3, 0.4], [0.0, 0.0, 0.5, 0.5]):          # tier level is the min
        cc = np.array([c], np.float32)
        np.testing.assert_allclose(oracle.cost_matrix_tiers(fanout, role, bw, lat, cc, 1e9),
                                   oracle.cost_matrix(fanout, role, bw, lat, cc[:, level], 1e9),
                                   rtol=1e-15)
    cc = np.array([[0.99, 0.0, 0.0, 0.0]], np.float32)                 # level 0 congested
    per_tier = oracle.cost_matrix_tiers(fanout, role, bw, lat, cc, 1e9)
    per_link = oracle.cost_matrix(fanout, role, bw, lat, cc[:, level], 1e9)
    taus = np.array([[tree.tier(p, d) for d in range(1, 16, 2)] for p in range(0, 16, 2)])
    assert (per_link[0][taus > 0] > per_tier[0][taus > 0]).all()      # the level-0 link binds
    np.testing.assert_array_equal(per_link[0][taus == 0], per_tier[0][taus == 0])
    one_minus_c = 1.0 - cc[0].astype(np.float64)
    np.testing.assert_allclose(per_tier[0], 1e9 / (np.array(bw)[taus] * one_minus_c[taus])
                               + np.array(lat)[taus], rtol=1e-15)


def test_per_tier_greedy_matches_exact_rational_bruteforce():
    theta = float(np.float32(1e-6))
    for seed in range(20):
        pb = _tiny_problem(seed)
        c = np.random.default_rng(1100 + seed).uniform(0, 0.9, size=(pb["u"].shape[0], 4)).astype(np.float32)
        w = tuple(float(np.float32(x)) for x in np.random.default_rng(1200 + seed).uniform(0, 2, 3))
        res = oracle.schedule_stream(pb["fanout"], pb["role"], pb["bw"], pb["lat"], c,
                                     pb["length"], pb["prefill"], pb["snap"], pb["M"], pb["events"],
                                     w[0], w[1], w[2], theta, pb["cap"], 81920, tier_mode=True)
        dec, best, load = naive.greedy_exact(pb["tree"], pb["role"], pb["bw"], pb["lat"], c,
                                             pb["length"], pb["prefill"], pb["snap"], pb["M"],
                                             pb["events"], w, theta, pb["cap"], 81920, tier_mode=True)
        assert list(res.dec) == dec and list(res.load) == load
        for r in range(len(dec)):
            if dec[r] >= 0:
                assert res.best[r] == pytest.approx(float(best[r]), rel=1e-14)


# ---------------------------------------- the paper's compute-load model (NEXT)
T_A, T_B = float(np.float32(0.012)), float(np.float32(0.0004))   # t_iter = a + b beta, seconds


def _run_load(pb, w, beta_max=4, m_min=0, m0=None, bpt=81920):
    m0 = pb["cap"] * bpt if m0 is None else m0
    return oracle.schedule_stream_load(pb["fanout"], pb["role"], pb["bw"], pb["lat"], pb["u"],
                                       pb["length"], pb["prefill"], pb["snap"], pb["M"],
                                       pb["events"], w[0], w[1], w[2], bpt, T_A, T_B, beta_max,
                                       m_min, m0)


def test_load_model_matches_exact_rational_bruteforce():
    n_cmp = 0
    for seed in range(40):
        pb = _tiny_problem(seed, R=10)
        w = tuple(float(np.float32(x)) for x in np.random.default_rng(1300 + seed).uniform(0, 2, 3))
        bmax, m_min = (2, 3, 64)[seed % 3], (0, 10 ** 8)[seed % 2]
        m0 = int(np.random.default_rng(seed).integers(2, 9)) * 10 ** 8
        res = _run_load(pb, w, bmax, m_min, m0)
        dec, best, n, m = naive.greedy_exact_load(pb["tree"], pb["role"], pb["bw"], pb["lat"],
                                                  pb["u"], pb["length"], pb["prefill"], pb["snap"],
                                                  pb["M"], pb["events"], w, 81920, T_A, T_B, bmax,
                                                  m_min, m0)
        assert list(res.dec) == dec and list(res.n) == n and list(res.m) == m
        for r in range(len(dec)):
            if dec[r] >= 0:
                assert res.best[r] == pytest.approx(float(best[r]), rel=1e-14)
                n_cmp += 1
    assert n_cmp > 150


def _one_decode_stream(R, beta_max, lengths=None, departures=()):
    """One prefill, one decode (instances 0 and 1 of a (2,1,1,1) tree), R arrivals in
    order, then the departures listed (request indices) in that order."""
    fanout = (2, 1, 1, 1)
    role = np.array([0, 1], np.uint8)
    L = oracle.used_links(fanout)
    length = np.full(R, 64, np.uint32) if lengths is None else np.asarray(lengths, np.uint32)
    events = list(range(R)) + [r | (1 << 31) for r in departures]
    return dict(fanout=fanout, role=role, bw=[900e9, 400e9, 200e9, 100e9], lat=[0.0] * 4,
                u=np.zeros((1, L), np.float32), length=length, prefill=np.zeros(R, np.uint32),
                snap=np.zeros(R, np.uint32), M=np.zeros((R, 1), np.uint16),
                events=np.array(events, np.uint32), cap=0)


def test_load_model_queue_and_decode_terms():
    """Sec. IV-B on one decode with beta_max = 4 and only the load term: the k-th arrival
    sees k requests; below beta_max it joins the batch (T_queue = 0, T_decode = a + b(k+1)),
    above it waits one iteration per blocked predecessor: T_queue = (k - 4)(a + 4b)."""
    R = 9
    res = _run_load(_one_decode_stream(R, 4), (0.0, 0.0, 1.0), beta_max=4, m0=10 ** 15)
    a, b = T_A, T_B
    for k in range(R):
        beta = min(k, 4)
        expect = max(0, k - 4) * (a + b * beta) + a + b * (beta + 1)
        assert res.best[k] == pytest.approx(expect, rel=1e-15)
    assert list(res.n) == [R]


def test_load_model_memory_filter():
    """Feasible iff m >= s_eff + m_min (the objective's feasible set, Sec. IV-A): with
    room for two requests' KV the third is rejected; a departure returns its bytes."""
    per = 64 * 81920                                  # 64 tokens, no prefix hit
    pb = _one_decode_stream(3, 64)
    res = _run_load(pb, (1.0, 1.0, 1.0), beta_max=64, m0=2 * per + 5, m_min=5)
    assert list(res.dec) == [0, 0, -1] and list(res.m) == [5]
    pb = _one_decode_stream(3, 64, departures=(0,))
    pb["events"] = np.array([0, 1, 0 | (1 << 31), 2], np.uint32)
    res = _run_load(pb, (1.0, 1.0, 1.0), beta_max=64, m0=2 * per + 5, m_min=5)
    assert list(res.dec) == [0, 0, 0] and list(res.n) == [2] and list(res.m) == [5]


# ------------------------------------------ evolving caches (NEXT: cache update on dispatch)
def _evolving_problem(seed, R=10, span=1000):
    """A tiny tree (P = D = 4) whose requests share three roots (random depths, tails of
    their own) and whose caches hold root prefixes with holes."""
    pb = _tiny_problem(seed, R=R, span=span)
    rng = np.random.default_rng(2000 + seed)
    roots = [rng.integers(1, 2 ** 63, 80, dtype=np.int64).astype(np.uint64) for _ in range(3)]
    chains = []
    for r in range(R):
        n = int(pb["length"][r]) // 16
        k = int(rng.integers(0, min(n, 80) + 1))
        c = np.concatenate([roots[int(rng.integers(0, 3))][:k],
                            rng.integers(1, 2 ** 63, n - k, dtype=np.int64).astype(np.uint64)])
        if r >= 2 and rng.random() < 0.3:              # a repeat of an earlier prefix
            prev = chains[int(rng.integers(0, r))]
            c = np.concatenate([prev[:min(len(prev), n)],
                                rng.integers(1, 2 ** 63, max(0, n - len(prev)), dtype=np.int64).astype(np.uint64)])
        chains.append(c.astype(np.uint64))
    D = int(pb["role"].sum())
    keys = []
    for d in range(D):
        ks = []
        for root in roots:
            depth = int(rng.integers(0, 81))
            keep = list(root[:depth])
            if depth > 5 and rng.random() < 0.3:
                keep.pop(int(rng.integers(0, depth)))
            ks += keep
        keys.append(np.array(ks, np.uint64))
    pb["chains"], pb["keys"] = chains, keys
    return pb


def _run_evolving(pb, w, theta=float(np.float32(1e-6)), bpt=81920, cap=None,
                  cap_blocks=oracle.UNBOUNDED):
    keys = np.concatenate([np.asarray(k, np.uint64) for k in pb["keys"]])
    key_off = np.concatenate([[0], np.cumsum([len(k) for k in pb["keys"]])]).astype(np.uint64)
    chains = np.concatenate([np.asarray(c, np.uint64) for c in pb["chains"]])
    chain_off = np.concatenate([[0], np.cumsum([len(c) for c in pb["chains"]])]).astype(np.uint64)
    return oracle.schedule_stream_evolving(pb["fanout"], pb["role"], pb["bw"], pb["lat"], pb["u"],
                                           pb["length"], pb["prefill"], pb["snap"], keys, key_off,
                                           chains, chain_off, pb["events"], w[0], w[1], w[2],
                                           theta, pb["cap"] if cap is None else cap, bpt,
                                           cap_blocks=cap_blocks)


def test_evolving_matches_exact_rational_bruteforce():
    theta = float(np.float32(1e-6))
    grew = 0
    for seed in range(30):
        pb = _evolving_problem(seed)
        w = tuple(float(np.float32(x)) for x in np.random.default_rng(1400 + seed).uniform(0, 2, 3))
        res = _run_evolving(pb, w)
        dec, best, load, M, _ = naive.greedy_exact_evolving(
            pb["tree"], pb["role"], pb["bw"], pb["lat"], pb["u"], pb["length"], pb["prefill"],
            pb["snap"], pb["keys"], pb["chains"], pb["events"], w, theta, pb["cap"], 81920)
        assert list(res.dec) == dec and list(res.load) == load
        np.testing.assert_array_equal(res.M, np.array(M, np.uint16))
        for r in range(len(dec)):
            if dec[r] >= 0:
                assert res.best[r] == pytest.approx(float(best[r]), rel=1e-14)
        # the static match of the same caches: evolving hits are never below it
        keys = np.concatenate(pb["keys"])
        key_off = np.concatenate([[0], np.cumsum([len(k) for k in pb["keys"]])]).astype(np.uint64)
        chains = np.concatenate(pb["chains"])
        chain_off = np.concatenate([[0], np.cumsum([len(c) for c in pb["chains"]])]).astype(np.uint64)
        static = oracle.prefix_match(keys, key_off, len(pb["keys"]), chains, chain_off,
                                     np.array([0, len(pb["chains"])], np.uint32))
        assert (res.M >= static).all()
        grew += int((res.M > static).sum())
    assert grew > 10


def test_evolving_without_dispatches_is_the_static_match():
    """Nothing fits (cap 0): no cache grows, every arrival sees the static hits."""
    pb = _evolving_problem(3)
    res = _run_evolving(pb, (1.0, 1.0, 1.0), cap=0)
    assert (res.dec == -1).all()
    keys = np.concatenate(pb["keys"])
    key_off = np.concatenate([[0], np.cumsum([len(k) for k in pb["keys"]])]).astype(np.uint64)
    chains = np.concatenate(pb["chains"])
    chain_off = np.concatenate([[0], np.cumsum([len(c) for c in pb["chains"]])]).astype(np.uint64)
    np.testing.assert_array_equal(res.M, oracle.prefix_match(keys, key_off, 4, chains, chain_off,
                                                             np.array([0, len(pb["chains"])], np.uint32)))


def test_evolving_dispatch_warms_its_decode():
    """Request 1 repeats request 0's chain: after request 0 goes to some decode, that
    decode holds the whole chain and request 1 hits all of it there, and only there."""
    pb = _evolving_problem(5, R=2)
    pb["chains"][1] = pb["chains"][0].copy()
    pb["length"][1] = pb["length"][0]
    pb["events"] = np.array([0, 1, 1 << 31, 1 | (1 << 31)], np.uint32)
    res = _run_evolving(pb, (1.0, 1.0, 0.0), cap=10 ** 9)
    d0 = int(res.dec[0])
    n = len(pb["chains"][0])
    assert d0 >= 0 and res.M[1, d0] == n
    assert all(res.M[1, d] == res.M[0, d] for d in range(4) if d != d0)


# ------------------------------------------ LRU-managed caches (Sec. VI-B simulator)
def test_evolving_lru_matches_exact_rational_bruteforce():
    """Caches of a few dozen to a few hundred blocks, so that dispatches evict: decisions,
    hits, final loads and the final recency lists equal the exact-rational evaluator's,
    which keeps each cache as a plain list (most recent first) rebuilt on every dispatch."""
    theta = float(np.float32(1e-6))
    changed = 0
    for seed in range(30):
        pb = _evolving_problem(seed, R=14)
        w = tuple(float(np.float32(x)) for x in np.random.default_rng(2400 + seed).uniform(0, 2, 3))
        cap_blocks = (40, 120, 300)[seed % 3]
        res = _run_evolving(pb, w, cap_blocks=cap_blocks)
        dec, best, load, M, caches = naive.greedy_exact_evolving(
            pb["tree"], pb["role"], pb["bw"], pb["lat"], pb["u"], pb["length"], pb["prefill"],
            pb["snap"], pb["keys"], pb["chains"], pb["events"], w, theta, pb["cap"], 81920,
            cap_blocks=cap_blocks)
        assert list(res.dec) == dec and list(res.load) == load
        np.testing.assert_array_equal(res.M, np.array(M, np.uint16))
        for d in range(len(caches)):
            assert [int(x) for x in res.caches[d]] == caches[d]
            assert len(caches[d]) <= cap_blocks
        for r in range(len(dec)):
            if dec[r] >= 0:
                assert res.best[r] == pytest.approx(float(best[r]), rel=1e-14)
        free = _run_evolving(pb, w)
        changed += int((free.M != res.M).sum() + (free.dec != res.dec).sum())
    assert changed > 20  # eviction changed hits or decisions


def _lru_case(keys, chains, lengths, cap_blocks, w=(0.0, 1.0, 0.0)):
    """Arrivals only, one per chain, on the 4-decode tiny tree; prefix-only weights make
    every candidate's score its missed fraction (ties to the lowest decode)."""
    pb = _tiny_problem(7, R=len(chains))
    pb["keys"] = [np.asarray(k, np.uint64) for k in keys]
    pb["chains"] = [np.asarray(c, np.uint64) for c in chains]
    pb["length"] = np.asarray(lengths, np.uint32)
    pb["events"] = np.arange(len(chains), dtype=np.uint32)
    pb["cap"] = 10 ** 9
    return _run_evolving(pb, w, cap_blocks=cap_blocks)


X = [1000 + i for i in range(10)]
Y = [2000 + i for i in range(8)]


def test_lru_eviction_changes_a_later_decision():
    """d0 holds X0..X9, d1 holds X0..X5, each decode keeps 12 blocks.  A (8 new blocks,
    no hits) goes to d0 (all tie); its blocks become d0's most recent and the 6 least
    recent, X4..X9, are evicted.  B = X0..X9 then hits 4 blocks on d0 and 6 on d1 and goes
    to d1, while without eviction it would hit all 10 on d0 and go there."""
    keys = [X, X[:6], [], []]
    res = _lru_case(keys, [Y, X], [128, 160], 12)
    assert list(res.dec) == [0, 1]
    assert list(res.M[1]) == [4, 6, 0, 0]
    assert [int(h) for h in res.caches[0]] == Y + X[:4]
    assert [int(h) for h in res.caches[1]] == X           # B's chain, X6..X9 inserted
    free = _lru_case(keys, [Y, X], [128, 160], oracle.UNBOUNDED)
    assert list(free.dec) == [0, 0] and list(free.M[1]) == [10, 6, 0, 0]


def test_lru_chain_tail_is_evicted_first():
    """A (C0..C9) to an empty d0, then B (4 new blocks) to d0 as well: d0 keeps 12 blocks,
    so C8 and C9, the least recent (a chain's blocks are used from its last block to its
    first), go; E = C0..C9 then hits 8 blocks on d0."""
    C = [3000 + i for i in range(10)]
    Dn = [4000 + i for i in range(4)]
    res = _lru_case([[], [], [], []], [C, Dn, C], [160, 64, 160], 12)
    assert list(res.dec[:2]) == [0, 0]
    assert int(res.M[2, 0]) == 8
    # E goes to d0 (8 hits) and refreshes the whole chain: C0..C9, then Dn0, Dn1
    assert [int(h) for h in res.caches[0]] == C + Dn[:2]


def test_lru_refresh_keeps_reused_blocks():
    """d0 holds Z0..Z5 (most recent) then X0..X5.  A = X0 X1 X2 W0 W1 W2 hits 3 blocks on
    d0 and goes there; its blocks become the most recent, so the 12-block cache evicts
    X3..X5 and keeps the refreshed X0..X2: B = X0..X5 then hits 3 blocks on d0."""
    Z = [5000 + i for i in range(6)]
    W = [6000 + i for i in range(3)]
    res = _lru_case([Z + X[:6], [], [], []], [X[:3] + W, X[:6]], [96, 96], 12)
    assert int(res.dec[0]) == 0 and int(res.M[0, 0]) == 3
    assert int(res.M[1, 0]) == 3
    assert [int(h) for h in res.caches[0]][:12] == X[:6] + W + Z[:3]


def test_lru_initial_list_cut_to_capacity():
    """A key list longer than the capacity keeps its most recent (first) entries; with no
    dispatch (nothing fits) the hits are the static match against those entries."""
    K = [7000 + i for i in range(20)]
    pb = _tiny_problem(11, R=1)
    pb["keys"] = [np.asarray(K, np.uint64)] * 4
    pb["chains"] = [np.asarray(K, np.uint64)]
    pb["length"] = np.array([320], np.uint32)
    pb["events"] = np.array([0], np.uint32)
    res = _run_evolving(pb, (1.0, 1.0, 1.0), cap=0, cap_blocks=12)
    assert int(res.dec[0]) == -1
    assert list(res.M[0]) == [12] * 4
    assert all([int(h) for h in c] == K[:12] for c in res.caches)
