"""Parity at the full sizes of the other workloads of the hot path.

* Oracle-build sweep: all 1,000 snapshots of the 2,048 x 8,192-pair matrix over
  24,576-link rows (67 GB of fp32 costs) in the launch configuration bench.py's sweep
  times; a million sampled entries, whole rows and columns checked against the oracle.
* Prefix-heavy long context (1,024 decodes, 2^20-block caches, 8,192-block chains) and the
  large cluster (4,096 decodes, 16 streams of 100,000 requests): every prefix hit, sampled
  hits against the oracle's matcher, whole streams of the greedy against the oracle.
"""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_common import check_stream, rel_close

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


def test_oracle_sweep_full_size():
    from paper_2606_03910_gb300 import netkv
    spec = synth.config3(1000)
    w = synth.make_workload(spec)
    util = w.util()
    topo = netkv.netkv_topology_create(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, w.L)
    _, P, D, _ = netkv.netkv_topology_query(topo)
    C = torch.empty((1000, P, D), dtype=torch.float32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    netkv.netkv_oracle_build(topo, torch.from_numpy(util).cuda(), 1000, spec.kv_bytes, C, None, st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    rng = np.random.default_rng(123)
    n = 1_000_000
    s = rng.integers(0, 1000, n); p = rng.integers(0, P, n); d = rng.integers(0, D, n)
    idx = torch.from_numpy(((s * P + p) * D + d).astype(np.int64)).cuda()
    got = C.view(-1)[idx].cpu().numpy()
    ref = oracle.cost_entries(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, util, s, p, d,
                              spec.kv_bytes)
    assert rel_close(got, ref).all()
    for ss, pp in ((0, 0), (999, P - 1), (500, 1234)):
        ref = oracle.cost_entries(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, util,
                                  np.full(D, ss), np.full(D, pp), np.arange(D), spec.kv_bytes)
        assert rel_close(C[ss, pp].cpu().numpy(), ref).all()
    ref = oracle.cost_entries(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, util,
                              np.full(P, 999), np.arange(P), np.full(P, D - 1), spec.kv_bytes)
    assert rel_close(C[999, :, D - 1].cpu().numpy(), ref).all()
    del C
    torch.cuda.empty_cache()


# ---------------------------------------------------------------------------------------
# Long-context and large-cluster workloads, set up exactly as bench.py sets them up.
# Their caches (1,024 x 2^20 and 4,096 x 200K blocks) are too large for the oracle's
# per-stream hash sets, so the prefix hits are checked three ways: every entry against the
# hits the generator constructs (pinned against the oracle on small cases), sampled
# (request, decode) pairs against the oracle's own matcher on the real key lists, and
# whole streams of the greedy against the oracle given the constructed hits.

def _setup(kind):
    import bench
    dev = torch.device("cuda", 0)
    spec = bench.workload_spec(kind, 0, 0)
    w, sc, x, out = bench.setup_workload(spec, dev)
    sc.step(x, out)
    torch.cuda.synchronize()
    return w, sc, x, out


def _check_all_hits(w, out, rows=1 << 15):
    dep = torch.from_numpy(w.depth[0].astype(np.int16)).cuda()          # [D, n_roots]
    shared = torch.from_numpy(w.shared.astype(np.int16)).cuda()
    root = torch.from_numpy(w.root.astype(np.int64)).cuda()
    assert w.n_sets == 1
    for r0 in range(0, w.R, rows):
        r1 = min(w.R, r0 + rows)
        exp = torch.minimum(shared[r0:r1, None], dep[:, root[r0:r1]].T)
        assert torch.equal(out.M[r0:r1], exp), f"prefix hits differ in rows [{r0}, {r1})"


def _check_sampled_hits(w, out, n_req, seed):
    rng = np.random.default_rng(seed)
    rs = np.unique(np.concatenate([[0, w.R - 1], rng.choice(w.R, n_req, replace=False)]))
    chains = np.concatenate([w.chains(int(r), int(r) + 1) for r in rs])
    lens = (w.chain_off[rs + 1] - w.chain_off[rs]).astype(np.uint64)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.uint64)
    M = out.M[torch.from_numpy(rs).cuda()].cpu().numpy().view(np.uint16)
    for d in sorted({0, 63, 64, w.D // 2, w.D - 1}):
        ref = oracle.prefix_match_one(w.keys(0, d), chains, off)
        np.testing.assert_array_equal(M[:, d], ref, err_msg=f"decode {d}")


@pytest.fixture(scope="class")
def longctx():
    r = _setup("longctx")
    yield r
    del r
    torch.cuda.empty_cache()


@pytest.fixture(scope="class")
def cluster():
    r = _setup("cluster")
    yield r
    del r
    torch.cuda.empty_cache()


class TestLongContext:
    """1,024 decodes caching 2^20 blocks, 64 streams x 256 requests of 8,192-block chains."""

    def test_status_and_shape(self, longctx):
        w, sc, x, out = longctx
        assert int(out.status.item()) == 0
        assert (x.R, sc.D, x.n_streams) == (16_384, 1024, 64)
        assert sc.log2_capacity == 27

    def test_all_hits_constructed(self, longctx):
        w, sc, x, out = longctx
        _check_all_hits(w, out)

    def test_sampled_hits_oracle(self, longctx):
        w, sc, x, out = longctx
        _check_sampled_hits(w, out, 48, 7)

    def test_streams_oracle(self, longctx):
        w, sc, x, out = longctx
        rng = np.random.default_rng(4)
        for s in [0, 63] + [int(v) for v in rng.choice(np.arange(1, 63), 2, replace=False)]:
            r0, r1 = int(w.req_off[s]), int(w.req_off[s + 1])
            check_stream(w, s, out, M_expect=synth.constructed_hits(w, r0, r1))

    def test_repeatable(self, longctx):
        w, sc, x, out = longctx
        dec, M = out.dec.clone(), out.M.clone()
        sc.step(x, out)
        torch.cuda.synchronize()
        assert torch.equal(out.dec, dec) and torch.equal(out.M, M)


class TestLargeCluster:
    """4,096 decodes sharing 200K-block caches, 16 streams x 100,000 requests."""

    def test_status_and_shape(self, cluster):
        w, sc, x, out = cluster
        assert int(out.status.item()) == 0
        assert (x.R, sc.D, x.n_streams) == (1_600_000, 4096, 16)

    def test_all_hits_constructed(self, cluster):
        w, sc, x, out = cluster
        _check_all_hits(w, out)

    def test_sampled_hits_oracle(self, cluster):
        w, sc, x, out = cluster
        _check_sampled_hits(w, out, 256, 8)

    def test_streams_oracle(self, cluster):
        w, sc, x, out = cluster
        for s in (0, 15):
            r0, r1 = int(w.req_off[s]), int(w.req_off[s + 1])
            res = check_stream(w, s, out, M_expect=synth.constructed_hits(w, r0, r1))
            assert res.near_ties <= 20

    def test_repeatable(self, cluster):
        w, sc, x, out = cluster
        dec, best = out.dec.clone(), out.best.clone()
        sc.step(x, out)
        torch.cuda.synchronize()
        assert torch.equal(out.dec, dec) and torch.equal(out.best, best)
