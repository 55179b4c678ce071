"""Parity at the benchmark's full size and launch configuration.

The 4,096-replica workload is set up exactly as bench.py sets it up (same
generator, cache index sizing, workspace and kernels, level bottlenecks taken from the
utilisation rows in the base-score pass); one step runs through the public pipeline, and whole sampled streams (first, last and three random ones)
are checked against the CPU oracle: prefix hits and decisions bit-exact (near-ties
replayed and counted), scores within 1e-5 relative, final loads exact, level
bottlenecks within 1e-5.  A second step must reproduce the first bit for bit.
"""
import numpy as np
import pytest

from tests.gpu_common import check_stream

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def fullsize():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import bench
    dev = torch.device("cuda", 0)
    w, sc, x, out = bench.setup_replicas(4096, 0, dev)
    sc.fuse_level_bottlenecks = True   # the bench's step: level bottlenecks in the base pass
    assert sc.fused(x)
    sc.step(x, out)
    sc.oracle_build(x, out)            # UB as well, for the level-bottleneck check
    torch.cuda.synchronize()
    yield w, sc, x, out
    del sc, x, out
    torch.cuda.empty_cache()


def test_bench_workload_sampled_streams(fullsize):
    w, sc, x, out = fullsize
    assert int(out.status.item()) == 0
    assert x.R == 4_096_000 and x.n_streams == 4096
    rng = np.random.default_rng(2024)
    streams = [0, 4095] + [int(s) for s in rng.choice(np.arange(1, 4095), 3, replace=False)]
    near = 0
    for s in streams:
        res = check_stream(w, s, out)
        near += res.near_ties
    assert near <= 5


def test_bench_workload_repeatable(fullsize):
    w, sc, x, out = fullsize
    dec, M, best = out.dec.clone(), out.M.clone(), out.best.clone()
    sc.step(x, out)
    torch.cuda.synchronize()
    assert torch.equal(out.dec, dec) and torch.equal(out.M, M) and torch.equal(out.best, best)


def test_bench_workload_with_self_contention(fullsize):
    """bench.py --inflight 16: the same workload and step with the self-contention greedy
    (counter cap 16, the paper's default); three whole streams against the oracle, which
    computes its own prefix hits from the key lists (equal to the GPU's bit for bit), with
    decisions and transfer times exact (near-ties and one-microsecond roundings replayed
    and counted), scores within 1e-5 and final loads exact."""
    import dataclasses
    import synth
    from oracle.workload import run_stream_inflight
    from tests.gpu_common import THETA, host, rel_close
    w, sc, x, out = fullsize
    x2 = dataclasses.replace(x, arrival_us=torch.from_numpy(w.arrival_us.astype(np.int64)).cuda())
    o = sc.alloc_outputs(x.n_snap, x.R, x.n_streams)
    sc.inflight_cap = 16               # not fused: the step builds UB for this walk
    try:
        sc.step(x2, o)
        torch.cuda.synchronize()
    finally:
        sc.inflight_cap = 0
    assert int(o.status.item()) == 0
    assert torch.equal(o.M, out.M)
    dec, xfer = host(o.dec), host(o.xfer_us)
    best, second, load = host(o.best), host(o.second), host(o.load_final)
    near = adopted = 0
    for s in (0, 2047, 4095):
        r0, r1 = int(w.req_off[s]), int(w.req_off[s + 1])
        # the oracle matches the stream's chains against its own cache sets
        res = run_stream_inflight(w, s, THETA, w.spec.cap_tokens, synth.BYTES_PER_TOKEN_SHARD, 16,
                                  hint=dec[r0:r1], xfer_hint=xfer[r0:r1])
        np.testing.assert_array_equal(host(o.M[r0:r1]).view(np.uint16), res.M)
        assert res.mismatches == 0 and res.xfer_mismatches == 0
        np.testing.assert_array_equal(res.dec, dec[r0:r1])
        np.testing.assert_array_equal(res.xfer_us, xfer[r0:r1])
        ev = w.events[w.event_off[s]:w.event_off[s + 1]]
        arr = (ev[(ev >> 31) == 0] & 0x7FFFFFFF).astype(np.int64) - r0
        assert rel_close(best[r0:r1][arr], res.best[arr]).all()
        assert rel_close(second[r0:r1][arr], res.second[arr]).all()
        np.testing.assert_array_equal(load[s], res.load)
        near += res.near_ties
        adopted += res.xfer_adopted
    assert near <= 5 and adopted <= 5
