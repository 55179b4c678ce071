"""Parity of the CUDA path (through the C ABI) with the CPU oracle.

Integer outputs (prefix hits, decisions, loads) must match bit for bit;
fp32 costs, bottlenecks and scores within 1e-5 relative; decisions may differ
only at near-ties (the GPU's choice scores within 1e-5 of the oracle's best),
which are counted and replayed.
"""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_common import THETA, check_stream, host, make_scorer, rel_close, run_gpu

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.init()


def nk():
    from paper_2606_03910_gb300 import netkv
    return netkv


def status_of(t):
    torch.cuda.synchronize()
    return int(t.item())


# ============================================================== oracle build
def _oracle_case(fanout, role, util, kv=10e9, bw=(900e9, 400e9, 200e9, 100e9),
                 lat=(1e-6, 3e-6, 6e-6, 10e-6)):
    netkv = nk()
    topo = netkv.netkv_topology_create(fanout, role, bw, lat, util.shape[1])
    N, P, D, _ = netkv.netkv_topology_query(topo)
    S = util.shape[0]
    du = torch.from_numpy(util).cuda()
    C = torch.full((S, P, D), -1.0, device="cuda")
    UB = torch.full((S, N, 4), -1.0, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    netkv.netkv_oracle_build(topo, du, S, kv, C, UB, st)
    assert status_of(st) == 0
    return host(C), host(UB), topo


@pytest.mark.parametrize("fanout,rule", [((2, 2, 2, 2), "alternate"),   # all four tiers, D % 4 == 0
                                          ((2, 2, 2, 2), "mod3"),        # P=6, D=10: scalar stores
                                          ((3, 5, 7, 11), "alternate"),  # D=577, odd, one chunk
                                          ((2, 8, 9, 13), "mod7")])      # D=1604: ragged 2nd chunk
def test_oracle_build_full_matrix(fanout, rule):
    n = int(np.prod(fanout))
    i = np.arange(n)
    role = {"alternate": i % 2 == 1, "mod3": i % 3 != 0, "mod7": i % 7 != 0}[rule].astype(np.uint8)
    L = oracle.used_links(fanout) + 3
    rng = np.random.default_rng(n)
    util = rng.uniform(0, 0.97, size=(3, L)).astype(np.float32)
    bw = (900e9, 400e9, 200e9, 100e9)
    lat = (1e-6, 3e-6, 6e-6, 10e-6)
    C, UB, _ = _oracle_case(fanout, role, util)
    Co = oracle.cost_matrix(fanout, role, bw, lat, util, 10e9)
    assert C.shape == Co.shape
    assert rel_close(C, Co).all()
    UBo = oracle.up_bottleneck(fanout, bw, util)
    assert rel_close(UB, UBo).all()


def test_oracle_build_sweep_shape_sampled():
    """2,048 x 8,192 pairs, 24,576-link Beta(2,5) + hot-link snapshots (3 snapshots):
    sampled entries, one full row and one full column against the oracle."""
    spec = synth.config3(n_snapshots=3)
    w = synth.make_workload(spec)
    util = w.util()
    C, UB, _ = _oracle_case(spec.fanout, w.role, util, kv=spec.kv_bytes)
    assert C.shape == (3, 2048, 8192)
    rng = np.random.default_rng(0)
    n = 200_000
    s = rng.integers(0, 3, n); p = rng.integers(0, 2048, n); d = rng.integers(0, 8192, n)
    ref = oracle.cost_entries(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, util, s, p, d,
                              spec.kv_bytes)
    assert rel_close(C[s, p, d], ref).all()
    for (ss, pp) in ((0, 0), (2, 2047)):
        dd = np.arange(8192)
        ref = oracle.cost_entries(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, util,
                                  np.full(8192, ss), np.full(8192, pp), dd, spec.kv_bytes)
        assert rel_close(C[ss, pp], ref).all()
    pp = np.arange(2048)
    ref = oracle.cost_entries(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, util,
                              np.full(2048, 1), pp, np.full(2048, 8191), spec.kv_bytes)
    assert rel_close(C[1, :, 8191], ref).all()
    UBo = oracle.up_bottleneck(spec.fanout, spec.tier_bw, util)
    assert rel_close(UB, UBo).all()


def test_oracle_build_edge_cases():
    netkv = nk()
    fanout = (2, 2, 2, 2)
    role = (np.arange(16) % 2).astype(np.uint8)
    L = oracle.used_links(fanout)
    topo = netkv.netkv_topology_create(fanout, role, (900e9, 400e9, 200e9, 100e9),
                                       (1e-6, 3e-6, 6e-6, 10e-6), L)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    u = torch.zeros((2, L), device="cuda")
    C = torch.empty((2, 8, 8), device="cuda")
    # nothing to do
    netkv.netkv_oracle_build(topo, u, 0, 1e9, C, None, st)
    # both outputs NULL, non-positive payload
    with pytest.raises(netkv.NetKVError):
        netkv.netkv_oracle_build(topo, u, 2, 1e9, None, None, st)
    with pytest.raises(netkv.NetKVError):
        netkv.netkv_oracle_build(topo, u, 2, 0.0, C, None, st)
    assert status_of(st) == 0
    # utilisation outside [0, 1) is reported, not trapped
    for bad in (1.0, float("nan"), -0.25):
        st.zero_()
        u2 = u.clone()
        u2[1, 3] = bad
        netkv.netkv_oracle_build(topo, u2, 2, 1e9, C, None, st)
        assert status_of(st) & netkv.NETKV_DEV_EDOMAIN
    # invalid topologies
    with pytest.raises(netkv.NetKVError):
        netkv.netkv_topology_create((2, 0, 2, 2), role, (1, 1, 1, 1), (0, 0, 0, 0), L)
    with pytest.raises(netkv.NetKVError):
        netkv.netkv_topology_create(fanout, np.zeros(16, np.uint8), (1, 1, 1, 1), (0, 0, 0, 0), L)
    with pytest.raises(netkv.NetKVError):
        netkv.netkv_topology_create(fanout, role, (1, 1, 1, 1), (0, 0, 0, 0), L - 1)


# ============================================================== prefix match
def _prefix_case(chains_list, caches, D, set_sizes, log2_cap=None):
    """caches[g][d] = list of keys; chains_list[r]; set_sizes = requests per set.
    log2_cap None: sized for load factor <= 0.5 per (set, group of 64 decodes)."""
    netkv = nk()
    if log2_cap is None:
        most = max(len(set().union(*[set(int(k) for k in caches[g][d]) for d in range(q, min(q + 64, D))]))
                   for g in range(len(set_sizes)) for q in range(0, D, 64))
        log2_cap = netkv.index_log2_capacity(most)
    n_sets = len(set_sizes)
    chains = np.concatenate([np.asarray(c, np.uint64) for c in chains_list]) if chains_list else np.zeros(0, np.uint64)
    chain_off = np.concatenate([[0], np.cumsum([len(c) for c in chains_list])]).astype(np.uint64)
    set_off = np.concatenate([[0], np.cumsum(set_sizes)]).astype(np.uint32)
    keys_l = [np.asarray(caches[g][d], np.uint64) for g in range(n_sets) for d in range(D)]
    keys = np.concatenate(keys_l) if keys_l else np.zeros(0, np.uint64)
    key_off = np.concatenate([[0], np.cumsum([len(k) for k in keys_l])]).astype(np.uint64)
    R = len(chains_list)
    tables = torch.empty(netkv.netkv_cache_index_bytes(n_sets, D, log2_cap) // 8,
                         dtype=torch.int64, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    dk = torch.from_numpy(keys.view(np.int64)).cuda() if len(keys) else torch.zeros(1, dtype=torch.int64, device="cuda")
    st_build = torch.zeros(1, dtype=torch.int32, device="cuda")
    netkv.netkv_cache_build(tables, n_sets, D, log2_cap, dk,
                            torch.from_numpy(key_off.view(np.int64)).cuda(), st_build)
    M = torch.full((max(R, 1), D), -1, dtype=torch.int16, device="cuda")
    dch = torch.from_numpy(chains.view(np.int64)).cuda() if len(chains) else torch.zeros(1, dtype=torch.int64, device="cuda")
    d_off = torch.from_numpy(chain_off.view(np.int64)).cuda()
    d_set = torch.from_numpy(set_off.view(np.int32)).cuda()
    netkv.netkv_prefix_match(tables, D, log2_cap, n_sets, dch, d_off, R, d_set, M, st)
    s = status_of(st)
    Mh = host(M).view(np.uint16)[:R]
    # the grouped (workspace) form gives the same result and the same status
    ws = torch.empty(max(netkv.netkv_prefix_match_workspace_size(R), 256), dtype=torch.uint8,
                     device="cuda")
    M2 = torch.full((max(R, 1), D), -1, dtype=torch.int16, device="cuda")
    st2 = torch.zeros(1, dtype=torch.int32, device="cuda")
    netkv.netkv_prefix_match(tables, D, log2_cap, n_sets, dch, d_off, R, d_set, M2, st2,
                             workspace=ws)
    assert status_of(st2) == s
    np.testing.assert_array_equal(host(M2).view(np.uint16)[:R], Mh)
    s |= status_of(st_build)
    Mo = oracle.prefix_match(keys, key_off, D, chains, chain_off, set_off) if R else Mh
    return Mh, Mo, s, tables


def test_prefix_match_random_ragged():
    """37 decodes (groups of 8 with a ragged last group), 3 table sets of unequal size,
    chains of length 0, 1, 31, 32, 33 ... with planted prefixes, holes and filler."""
    rng = np.random.default_rng(5)
    D = 37
    set_sizes = [20, 1, 29]
    lengths = [0, 1, 31, 32, 33, 64, 65, 300, 257] + list(rng.integers(0, 400, sum(set_sizes) - 9))
    chains_list = [rng.integers(1, 2 ** 63, n, dtype=np.int64).astype(np.uint64) for n in lengths]
    caches = []
    r = 0
    for g, sz in enumerate(set_sizes):
        cg = []
        members = chains_list[r:r + sz]
        for d in range(D):
            ks = set(int(x) for x in rng.integers(1, 2 ** 63, 50, dtype=np.int64))
            for c in members:
                if len(c) == 0:
                    continue
                depth = int(rng.integers(0, len(c) + 1))
                ks.update(int(x) for x in c[:depth])
                if rng.random() < 0.3 and depth < len(c):   # a hole: later blocks cached
                    ks.update(int(x) for x in c[depth + 1:depth + 20])
            cg.append(sorted(ks))
        caches.append(cg)
        r += sz
    M, Mo, s, _ = _prefix_case(chains_list, caches, D, set_sizes)
    assert s == 0
    np.testing.assert_array_equal(M, Mo)
    assert (Mo > 0).mean() > 0.3


def test_prefix_match_shared_prefixes():
    """Trie-shaped requests: several roots, random-depth root prefixes with random tails,
    exact duplicates, chains that are prefixes of other chains, the same first block in
    different table sets, empty chains; caches hold root prefixes with holes."""
    rng = np.random.default_rng(11)
    D, set_sizes = 13, [60, 45, 1, 30]
    roots = [rng.integers(1, 2 ** 63, 700, dtype=np.int64).astype(np.uint64) for _ in range(5)]
    chains_list = []
    for g, sz in enumerate(set_sizes):
        for i in range(sz):
            kind = rng.integers(0, 6)
            root = roots[rng.integers(0, 5)]
            if kind == 0:
                c = np.zeros(0, np.uint64)
            elif kind == 1 and chains_list:
                c = chains_list[int(rng.integers(0, len(chains_list)))].copy()     # duplicate
            elif kind == 2 and chains_list:
                c0 = chains_list[int(rng.integers(0, len(chains_list)))]
                c = c0[:int(rng.integers(0, len(c0) + 1))].copy()                 # a prefix
            else:
                k = int(rng.integers(0, 700))
                tail = rng.integers(1, 2 ** 63, int(rng.integers(0, 80)), dtype=np.int64).astype(np.uint64)
                c = np.concatenate([root[:k], tail])
            chains_list.append(c)
    caches = []
    for g in range(len(set_sizes)):
        cg = []
        for d in range(D):
            ks = set(int(x) for x in rng.integers(1, 2 ** 63, 30, dtype=np.int64))
            for root in roots:
                depth = int(rng.integers(0, 701))
                keep = root[:depth]
                if rng.random() < 0.3 and depth > 10:                           # a hole
                    keep = np.delete(keep, int(rng.integers(0, depth)))
                ks.update(int(x) for x in keep)
            cg.append(sorted(ks))
        caches.append(cg)
    M, Mo, s, _ = _prefix_case(chains_list, caches, D, set_sizes)
    assert s == 0
    np.testing.assert_array_equal(M, Mo)
    assert (Mo > 50).mean() > 0.2


@pytest.mark.parametrize("D", [65, 200, 2112, 2113])
def test_prefix_match_shared_prefixes_wide(D):
    """Pools of several 64-decode groups (ragged last group; 33 and 34 groups at D = 2112
    and 2113, more than one warp of pending probes, in the 16-byte row form and the
    scalar one): trie-shaped requests with duplicates and prefixes
    of other chains; caches hold root prefixes with holes and, on some decodes, the first
    blocks of request chains, so members resume past the leader and find blocks there."""
    rng = np.random.default_rng(D)
    set_sizes = [40, 1, 25]
    roots = [rng.integers(1, 2 ** 63, 300, dtype=np.int64).astype(np.uint64) for _ in range(3)]
    chains_list = []
    for g, sz in enumerate(set_sizes):
        for i in range(sz):
            kind = rng.integers(0, 6)
            root = roots[rng.integers(0, 3)]
            if kind == 0:
                c = np.zeros(0, np.uint64)
            elif kind == 1 and chains_list:
                c = chains_list[int(rng.integers(0, len(chains_list)))].copy()
            elif kind == 2 and chains_list:
                c0 = chains_list[int(rng.integers(0, len(chains_list)))]
                c = c0[:int(rng.integers(0, len(c0) + 1))].copy()
            else:
                k = int(rng.integers(0, 301))
                tail = rng.integers(1, 2 ** 63, int(rng.integers(0, 40)), dtype=np.int64).astype(np.uint64)
                c = np.concatenate([root[:k], tail])
            chains_list.append(c)
    caches = []
    r0 = 0
    for g, sz in enumerate(set_sizes):
        members = chains_list[r0:r0 + sz]
        r0 += sz
        cg = []
        for d in range(D):
            ks = set(int(x) for x in rng.integers(1, 2 ** 63, 8, dtype=np.int64))
            for root in roots:
                depth = int(rng.integers(0, 301))
                keep = root[:depth]
                if rng.random() < 0.3 and depth > 10:
                    keep = np.delete(keep, int(rng.integers(0, depth)))
                ks.update(int(x) for x in keep)
            if rng.random() < 0.2:                     # leading blocks of a few whole chains
                for c in (members[int(j)] for j in rng.integers(0, sz, 2)):
                    ks.update(int(x) for x in c[:int(rng.integers(0, len(c) + 1))])
            cg.append(sorted(ks))
        caches.append(cg)
    M, Mo, s, _ = _prefix_case(chains_list, caches, D, set_sizes)
    assert s == 0
    np.testing.assert_array_equal(M, Mo)
    assert (Mo > 20).mean() > 0.1


def test_prefix_match_workspace_checks():
    netkv = nk()
    tables = torch.zeros(netkv.netkv_cache_index_bytes(1, 4, 4) // 8, dtype=torch.int64,
                         device="cuda")
    off = torch.tensor([0, 2], dtype=torch.int64, device="cuda")
    ch = torch.tensor([5, 6], dtype=torch.int64, device="cuda")
    M = torch.empty((1, 4), dtype=torch.int16, device="cuda")
    need = netkv.netkv_prefix_match_workspace_size(1)
    assert need > 0 and netkv.netkv_prefix_match_workspace_size(0) == 0
    small = torch.empty(need - 1, dtype=torch.uint8, device="cuda")
    with pytest.raises(netkv.NetKVError):
        netkv.netkv_prefix_match(tables, 4, 4, 1, ch, off, 1, None, M, None, workspace=small)
    big = torch.empty(need + 512, dtype=torch.uint8, device="cuda")
    with pytest.raises(netkv.NetKVError):         # not 256-byte aligned
        netkv.netkv_prefix_match(tables, 4, 4, 1, ch, off, 1, None, M, None,
                                 workspace=big[8:])
    netkv.netkv_prefix_match(tables, 4, 4, 1, ch, off, 1, None, M, None, workspace=big)
    torch.cuda.synchronize()
    assert (host(M) == 0).all()


def test_prefix_match_holes_and_duplicates():
    chains_list = [[1, 2, 3, 4, 5], [1, 2, 3], [9, 2, 3]]
    caches = [[[1, 2, 4, 5, 5, 5], [1, 2, 3, 4, 5, 1]], [[2, 3, 9, 9], [9, 3]]]
    M, Mo, s, _ = _prefix_case(chains_list, caches, 2, [2, 1], log2_cap=4)
    assert s == 0
    np.testing.assert_array_equal(M, np.array([[2, 5], [2, 3], [3, 1]], np.uint16))
    np.testing.assert_array_equal(M, Mo)


def test_prefix_match_full_table_and_bad_hashes():
    netkv = nk()
    # 20 distinct keys into 16 slots: EFULL, and probes of absent keys stay bounded
    keys = list(range(1, 21))
    chains_list = [[1, 2, 3], [100, 1], [0, 1]]
    M, _, s, _ = _prefix_case(chains_list, [[keys]], 1, [3], log2_cap=4)
    assert s & netkv.NETKV_DEV_EFULL
    assert s & netkv.NETKV_DEV_EDOMAIN          # the zero hash in the last chain
    assert M[1, 0] == 0 and M[2, 0] == 0
    # a zero key in a key list is reported and skipped
    M, Mo, s, _ = _prefix_case([[5, 6]], [[[0, 5, 6]]], 1, [1], log2_cap=4)
    assert s & netkv.NETKV_DEV_EDOMAIN and M[0, 0] == 2


def test_prefix_match_long_chain_saturates():
    netkv = nk()
    n = 70_000
    chain = np.arange(1, n + 1, dtype=np.uint64)
    M, _, s, _ = _prefix_case([chain], [[chain]], 1, [1], log2_cap=18)
    assert s & netkv.NETKV_DEV_EDOMAIN
    assert M[0, 0] == 65535


def test_prefix_match_empty_inputs():
    netkv = nk()
    tables = torch.empty(netkv.netkv_cache_index_bytes(1, 4, 4) // 8, dtype=torch.int64,
                         device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    off = torch.zeros(5, dtype=torch.int64, device="cuda")
    netkv.netkv_cache_build(tables, 1, 4, 4, None, off, st)    # clear only
    assert (host(tables) == 0).all()
    M = torch.empty((1, 4), dtype=torch.int16, device="cuda")
    netkv.netkv_prefix_match(tables, 4, 4, 1, None, off, 0, None, M, st)   # R = 0
    with pytest.raises(netkv.NetKVError):
        netkv.netkv_prefix_match(tables, 4, 0, 1, None, off, 1, None, M, st)
    with pytest.raises(netkv.NetKVError):
        netkv.netkv_prefix_match(tables, 4, 4, 2, None, off, 1, None, M, st)   # no set offsets
    assert status_of(st) == 0


# ============================================================== whole path per stream
def test_tiny_workload_all_tiers():
    w = synth.make_workload(synth.tiny_spec())
    _, x, out = run_gpu(w)
    assert status_of(out.status) == 0
    for s in range(w.n_streams):
        check_stream(w, s, out)


def test_tiny_workload_with_rejects():
    spec = synth.tiny_spec(cap_tokens=3000, len_median=1500)
    w = synth.make_workload(spec)
    _, x, out = run_gpu(w, cap=spec.cap_tokens)
    rej = 0
    for s in range(w.n_streams):
        res = check_stream(w, s, out, cap=spec.cap_tokens)
        rej += res.rejects
    assert rej > 0
    r = np.flatnonzero(host(out.dec) == -1)
    assert np.isinf(host(out.best)[r]).all() and np.isinf(host(out.second)[r]).all()


def test_single_stream_64gpu_full():
    """The single-stream 64-GPU workload: 1,000 requests, 8 decode caches of 200K blocks."""
    w = synth.make_workload(synth.config0())
    _, x, out = run_gpu(w)
    assert status_of(out.status) == 0
    res = check_stream(w, 0, out)
    assert res.rejects == 0


@pytest.mark.parametrize("fanout,rule,D", [((1, 8, 8, 5), "mod5", 256),    # 256 threads, 1 each
                                           ((1, 8, 8, 20), "mod5", 1024),  # 256 threads, 4 each
                                           ((3, 5, 7, 11), "alternate", 577),
                                           ((1, 8, 8, 80), "mod5", 4096),  # 1024 threads, 4 each
                                           ((1, 2, 3, 5), "alternate", 15),
                                           ((2, 3, 4, 2), "alternate", 24),  # one warp, 1 each
                                           ((1, 5, 5, 5), "mod5", 100),      # 256 threads, ragged
                                           ((1, 7, 11, 17), "mod5", 1047)])  # 512 threads, 4 each
def test_schedule_block_shapes(fanout, rule, D):
    spec = synth.Spec(name="shape", fanout=fanout, role_rule=rule, n_streams=2,
                      requests_per_stream=120, rate_per_s=40.0, len_median=2048.0,
                      len_clip=(16, 16384), n_roots=6, root_blocks=(1024,), n_keys=2000,
                      log2_cap=12, tables="shared", telemetry="shared", cap_tokens=60_000)
    w = synth.make_workload(spec)
    assert w.D == D
    _, x, out = run_gpu(w, cap=spec.cap_tokens)
    assert status_of(out.status) == 0
    for s in range(w.n_streams):
        check_stream(w, s, out, cap=spec.cap_tokens)


def test_reductions_on_gpu():
    """Zero network weight, zero network and prefix weight, all zero: ties are exact on
    both sides and must break to the lowest decode rank."""
    from paper_2606_03910_gb300.pipeline import weights_tensor
    spec = synth.tiny_spec(requests_per_stream=60)
    w = synth.make_workload(spec)
    for wt in ((0.0, 1.0, 1.0), (0.0, 0.0, 1.0), (0.0, 0.0, 0.0), (0.0, 1.0, 0.0)):
        w.weights[:] = np.array(wt, np.float32)
        _, x, out = run_gpu(w)
        for s in range(w.n_streams):
            res = check_stream(w, s, out)
            if wt != (0.0, 1.0, 1.0):      # exact ties in both precisions
                assert res.near_ties == 0


def test_resume_from_load_init():
    """Splitting a stream's events in two calls, the second starting from the first's
    final loads, gives the same decisions and loads as one call."""
    import dataclasses
    w = synth.make_workload(synth.tiny_spec(n_streams=1, requests_per_stream=80))
    sc, x, out = run_gpu(w)
    E = int(w.event_off[-1])
    half = E // 2
    x1 = dataclasses.replace(x, event_off=torch.tensor([0, half], dtype=torch.int64, device="cuda"))
    o1 = sc.alloc_outputs(x.n_snap, x.R, 1)
    sc.step(x1, o1)
    x2 = dataclasses.replace(x, events=x.events[half:].contiguous(),
                             event_off=torch.tensor([0, E - half], dtype=torch.int64, device="cuda"),
                             load_init=o1.load_final.clone())
    o2 = dataclasses.replace(sc.alloc_outputs(x.n_snap, x.R, 1), UB=out.UB, M=out.M)
    o2.dec.copy_(o1.dec)
    sc.schedule(x2, o2)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(host(o2.load_final), host(out.load_final))
    ev = w.events[half:]
    arr = (ev[(ev >> 31) == 0] & 0x7FFFFFFF).astype(np.int64)
    np.testing.assert_array_equal(host(o2.dec)[arr], host(out.dec)[arr])


def test_schedule_edge_cases():
    netkv = nk()
    from paper_2606_03910_gb300.pipeline import weights_tensor
    w = synth.make_workload(synth.tiny_spec(n_streams=1, requests_per_stream=10))
    sc, x, out = run_gpu(w)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    # zero streams: nothing to do
    netkv.netkv_schedule_streams(sc.topo, 0, x.weights, x.R, x.length, x.prefill, x.snap, out.M,
                                 out.UB, x.n_snap, x.events, x.event_off, None, out.dec, out.best,
                                 out.second, out.load_final, st)
    # an empty event list leaves the initial loads
    eo = torch.zeros(2, dtype=torch.int64, device="cuda")
    li = torch.arange(8, dtype=torch.int64, device="cuda").reshape(1, 8)
    lf = torch.empty_like(li)
    netkv.netkv_schedule_streams(sc.topo, 1, x.weights, x.R, x.length, x.prefill, x.snap, out.M,
                                 out.UB, x.n_snap, x.events, eo, li, out.dec, out.best, out.second,
                                 lf, st)
    assert status_of(st) == 0
    np.testing.assert_array_equal(host(lf), host(li))
    # out-of-range snapshot and request indices, zero-length request: flagged, skipped
    bad_snap = x.snap.clone(); bad_snap[0] = x.n_snap + 5
    netkv.netkv_schedule_streams(sc.topo, 1, x.weights, x.R, x.length, x.prefill, bad_snap, out.M,
                                 out.UB, x.n_snap, x.events, x.event_off, None, out.dec, out.best,
                                 out.second, lf, st)
    assert status_of(st) & netkv.NETKV_DEV_ERANGE
    st.zero_()
    bad_len = x.length.clone(); bad_len[1] = 0
    netkv.netkv_schedule_streams(sc.topo, 1, x.weights, x.R, bad_len, x.prefill, x.snap, out.M,
                                 out.UB, x.n_snap, x.events, x.event_off, None, out.dec, out.best,
                                 out.second, lf, st)
    assert status_of(st) & netkv.NETKV_DEV_EDOMAIN
    assert int(host(out.dec)[1]) == -1
    st.zero_()
    bad_ev = x.events.clone(); bad_ev[0] = 0x7FFFFFF0
    netkv.netkv_schedule_streams(sc.topo, 1, x.weights, x.R, x.length, x.prefill, x.snap, out.M,
                                 out.UB, x.n_snap, bad_ev, x.event_off, None, out.dec, out.best,
                                 out.second, lf, st)
    assert status_of(st) & netkv.NETKV_DEV_ERANGE
    with pytest.raises(netkv.NetKVError):
        netkv.netkv_schedule_streams(sc.topo, 1, None, x.R, x.length, x.prefill, x.snap, out.M,
                                     out.UB, x.n_snap, x.events, x.event_off, None, out.dec,
                                     out.best, out.second, lf, st)


def test_copy_async_host_and_device():
    """Kernel copies between pinned host and device memory, including ragged tails."""
    netkv = nk()
    gen = torch.Generator().manual_seed(3)
    for nbytes in (16, 17, 4096 + 5, 3 * 2 ** 20 + 15):
        h = torch.randint(0, 255, (nbytes,), dtype=torch.uint8, generator=gen).pin_memory()
        d = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
        netkv.netkv_copy_async(d, h, nbytes)
        d2 = torch.zeros_like(d)
        netkv.netkv_copy_async(d2, d, nbytes)
        h2 = torch.zeros(nbytes, dtype=torch.uint8).pin_memory()
        netkv.netkv_copy_async(h2, d2, nbytes)
        torch.cuda.synchronize()
        assert torch.equal(d.cpu(), h) and torch.equal(h2, h)
    netkv.netkv_copy_async(d, h, 0)                      # nothing to do
    with pytest.raises(netkv.NetKVError):
        netkv.netkv_copy_async(d[1:], h, 16)             # misaligned destination


def test_index_key_order_does_not_change_results():
    """The same caches listed in chain order (long runs) and shuffled (no runs) give the
    same prefix hits; chain order is only faster."""
    from synth import stage
    netkv = nk()
    w = synth.make_workload(synth.config0())
    from tests.gpu_common import index_log2
    L = index_log2(w)
    keys = stage.keys(w, 0, w.n_sets)
    key_off = stage.key_offsets(w, w.n_sets * w.D)
    ra = stage.request_arrays(w)
    chains = stage.chains(w)
    Ms = []
    for shuffle in (False, True):
        k = keys.clone()
        if shuffle:
            ko = key_off.cpu().numpy()
            for t in range(w.D):
                seg = k[ko[t]:ko[t + 1]]
                k[ko[t]:ko[t + 1]] = seg[torch.randperm(seg.numel(), device=seg.device)]
        index = torch.empty(netkv.netkv_cache_index_bytes(1, w.D, L) // 8, dtype=torch.int64,
                            device="cuda")
        st = torch.zeros(1, dtype=torch.int32, device="cuda")
        netkv.netkv_cache_build(index, 1, w.D, L, k, key_off, st)
        M = torch.empty((w.R, w.D), dtype=torch.int16, device="cuda")
        netkv.netkv_prefix_match(index, w.D, L, 1, chains, ra["chain_off"], w.R, None, M, st)
        assert status_of(st) == 0
        Ms.append(M)
    assert torch.equal(Ms[0], Ms[1])
    assert (host(Ms[0]).view(np.uint16) > 100).any()


@pytest.mark.parametrize("make_spec", [synth.tiny_spec, synth.config0])
def test_greedy_without_workspace(make_spec):
    """The fused greedy (no base-score workspace) against the oracle."""
    w = synth.make_workload(make_spec())
    sc = make_scorer(w)
    sc.precompute_scores = False
    _, x, out = run_gpu(w, sc=sc)
    assert status_of(out.status) == 0
    for s in range(w.n_streams):
        check_stream(w, s, out)


@pytest.mark.parametrize("zero_copy", [(), ("chains",)])
def test_host_buffer_step(zero_copy):
    """The step from pinned host buffers (copied, or chains read in place over the
    host link) gives exactly the device-resident step's results."""
    import dataclasses
    from paper_2606_03910_gb300.pipeline import StepInputs
    w = synth.make_workload(synth.config0())
    sc, x, out = run_gpu(w)
    ref = {k: getattr(out, k).clone() for k in ("dec", "best", "second", "load_final", "M")}
    xh = StepInputs(**{f.name: (getattr(x, f.name).cpu().pin_memory()
                                if isinstance(getattr(x, f.name), torch.Tensor) else None)
                       for f in dataclasses.fields(StepInputs)})
    xd = StepInputs(**{f.name: (torch.empty_like(getattr(x, f.name))
                                if isinstance(getattr(x, f.name), torch.Tensor) else None)
                       for f in dataclasses.fields(StepInputs)})
    out2 = sc.alloc_outputs(x.n_snap, x.R, x.n_streams)
    res_h = {k: torch.empty_like(getattr(out, k), device="cpu").pin_memory()
             for k in ("dec", "best", "second", "load_final")}
    sc.step_host(xh, xd, out2, res_h, zero_copy=zero_copy)
    torch.cuda.synchronize()
    assert status_of(out2.status) == 0
    for k in ("dec", "best", "second", "load_final"):
        assert torch.equal(res_h[k], ref[k].cpu()), k
    assert torch.equal(out2.M, ref["M"])
