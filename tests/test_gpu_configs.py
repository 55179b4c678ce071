"""Parity at the full sizes of the other workloads of the hot path.

* Oracle-build sweep: all 1,000 snapshots of the 2,048 x 8,192-pair matrix over
  24,576-link rows (67 GB of fp32 costs) in the launch configuration bench.py's sweep
  times; a million sampled entries, whole rows and columns checked against the oracle.
"""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_common import rel_close

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
