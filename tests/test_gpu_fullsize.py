"""Parity at the benchmark's full size and launch configuration.

The 4,096-replica workload is set up exactly as bench.py sets it up (same
generator, cache index sizing, workspace and kernels); one step runs through the
public pipeline, and whole sampled streams (first, last and three random ones)
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
    sc.step(x, out)
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
