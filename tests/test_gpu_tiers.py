"""GPU parity of the paper-literal per-tier oracle (netkv_oracle_build_tiers: the tier,
bandwidth, congestion and latency maps of Sec. III-E, a pair's bandwidth B_tau (1 - c_tau))
against the oracle.

* Every entry of C and of UB within 1e-5 of the oracle's per-tier matrix and maps, on
  trees where every tier occurs, odd and ragged decode counts.
* The worked example of Sec. III-D through the library.
* The whole step with per-tier maps on the tiny workload and every greedy launch shape:
  whole streams against the oracle's per-tier greedy.
"""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_common import check_stream, host, rel_close, run_gpu

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


def nk():
    from paper_2606_03910_gb300 import netkv
    return netkv


@pytest.mark.parametrize("fanout,k", [((2, 2, 2, 2), 2), ((2, 2, 2, 2), 3), ((3, 5, 7, 11), 2),
                                      ((2, 8, 9, 13), 7)])
def test_tiers_oracle_build(fanout, k):
    netkv = nk()
    n = int(np.prod(fanout))
    role = (np.arange(n) % k != 0).astype(np.uint8)
    L = oracle.used_links(fanout)
    bw, lat = (900e9, 400e9, 200e9, 100e9), (1e-6, 3e-6, 6e-6, 10e-6)
    S = 3
    c = np.random.default_rng(n).uniform(0, 0.95, size=(S, 4)).astype(np.float32)
    topo = netkv.netkv_topology_create(fanout, role, bw, lat, L)
    _, P, D, _ = netkv.netkv_topology_query(topo)
    C = torch.empty((S, P, D), dtype=torch.float32, device="cuda")
    UB = torch.empty((S, n, 4), dtype=torch.float32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    netkv.netkv_oracle_build_tiers(topo, torch.from_numpy(c).cuda(), S, 2.5e9, C, UB, st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert rel_close(host(C), oracle.cost_matrix_tiers(fanout, role, bw, lat, c, 2.5e9)).all()
    per_tier = np.asarray(bw) * (1.0 - c.astype(np.float64))
    assert rel_close(host(UB), np.repeat(per_tier[:, None, :], n, axis=1)).all()


def test_tiers_worked_example():
    """Sec. III-D: d1 (tier 2) at B2 (1 - c) = 5 GB/s, d2 (tier 3) at 2.5 GB/s, and 1.5625
    GB/s with c3 = 0.5; costs of 1 GB and 5 GB transfers."""
    netkv = nk()
    fanout = (2, 2, 2, 2)
    role = np.zeros(16, np.uint8)
    role[[4, 8]] = 1
    topo = netkv.netkv_topology_create(fanout, role, (100e9, 50e9, 6.25e9, 3.125e9),
                                       (0.0,) * 4, oracle.used_links(fanout))
    c = torch.tensor([[0.2, 0.2, 0.2, 0.2], [0.2, 0.2, 0.2, 0.5]], dtype=torch.float32,
                     device="cuda")
    C = torch.empty((2, 14, 2), dtype=torch.float32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    netkv.netkv_oracle_build_tiers(topo, c, 2, 1e9, C, None, st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert float(C[0, 0, 0]) == pytest.approx(0.2, rel=1e-6)     # 1 GB at 5 GB/s
    assert float(C[0, 0, 1]) == pytest.approx(0.4, rel=1e-6)     # 1 GB at 2.5 GB/s
    assert float(C[1, 0, 1]) == pytest.approx(0.64, rel=1e-6)    # 1 GB at 1.5625 GB/s


@pytest.mark.parametrize("fanout,rule,D", [((2, 2, 2, 2), "alternate", 8),
                                           ((1, 2, 3, 5), "alternate", 15),
                                           ((2, 3, 4, 2), "alternate", 24),
                                           ((1, 5, 5, 5), "mod5", 100),
                                           ((3, 5, 7, 11), "alternate", 577),
                                           ((1, 8, 8, 80), "mod5", 4096)])
def test_tiers_step_streams(fanout, rule, D):
    spec = synth.Spec(name="tiers", fanout=fanout, role_rule=rule, n_streams=2,
                      requests_per_stream=120, rate_per_s=40.0, len_median=2048.0,
                      len_clip=(16, 16384), n_roots=6, root_blocks=(1024,), n_keys=2000,
                      log2_cap=12, tables="shared", telemetry="shared", cap_tokens=60_000)
    w = synth.make_workload(spec)
    assert w.D == D
    _, x, out = run_gpu(w, cap=spec.cap_tokens, tiers=True)
    assert int(out.status.item()) == 0
    near = 0
    for s in range(w.n_streams):
        near += check_stream(w, s, out, cap=spec.cap_tokens, tiers=True).near_ties
    assert near <= 3
