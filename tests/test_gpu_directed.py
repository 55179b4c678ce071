"""GPU parity of directed links (netkv_oracle_build_directed: one utilisation per link
and direction, a transfer climbing the prefill's links upward and descending the
decode's downward) against the oracle.

* Equal upward and downward rows give netkv_oracle_build's C and UB bit for bit.
* Distinct rows: every entry of C and UB within 1e-5 of the oracle's directed matrix
  and level bottlenecks, on trees where every tier occurs, odd and ragged decode counts.
* The whole step (level bottlenecks, prefix match, greedy) with directed rows on the
  tiny workload and every greedy launch shape: whole streams against the oracle's
  directed greedy (prefix hits and decisions exact, near-ties replayed and counted,
  scores within 1e-5).
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


SHAPES = [((2, 2, 2, 2), 2),     # prefill iff i % 2 == 0: P = D = 8, every tier
          ((2, 2, 2, 2), 3),     # P = 6, D = 10: scalar stores
          ((3, 5, 7, 11), 2),    # D = 577, odd
          ((2, 8, 9, 13), 7)]    # D = 1,604: ragged second chunk


@pytest.mark.parametrize("fanout,k", SHAPES)
def test_directed_oracle_build(fanout, k):
    netkv = nk()
    n = int(np.prod(fanout))
    role = (np.arange(n) % k != 0).astype(np.uint8)
    L = oracle.used_links(fanout) + 3
    bw, lat = (900e9, 400e9, 200e9, 100e9), (1e-6, 3e-6, 6e-6, 10e-6)
    rng = np.random.default_rng(sum(fanout))
    S = 2
    up = rng.uniform(0, 0.95, size=(S, L)).astype(np.float32)
    down = rng.uniform(0, 0.95, size=(S, L)).astype(np.float32)
    topo = netkv.netkv_topology_create(fanout, role, bw, lat, L)
    _, P, D, _ = netkv.netkv_topology_query(topo)
    N = P + D
    dev = lambda a: torch.from_numpy(a).cuda()
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    # equal rows: the undirected call, bit for bit
    C0 = torch.empty((S, P, D), dtype=torch.float32, device="cuda")
    U0 = torch.empty((S, N, 4), dtype=torch.float32, device="cuda")
    netkv.netkv_oracle_build(topo, dev(up), S, 2.5e9, C0, U0, st)
    C1, U1 = torch.empty_like(C0), torch.empty_like(U0)
    netkv.netkv_oracle_build_directed(topo, dev(up), dev(up), S, 2.5e9, C1, U1, st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert torch.equal(C0, C1) and torch.equal(U0, U1)
    # distinct rows against the oracle
    netkv.netkv_oracle_build_directed(topo, dev(up), dev(down), S, 2.5e9, C1, U1, st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    ref_C = oracle.cost_matrix_directed(fanout, role, bw, lat, up, down, 2.5e9)
    ref_U = oracle.level_bottleneck_directed(fanout, role, bw, up, down)
    assert rel_close(host(C1), ref_C).all()
    assert rel_close(host(U1), ref_U).all()
    assert not torch.equal(C0, C1)      # the downward rows matter


@pytest.mark.parametrize("fanout,rule,D", [((2, 2, 2, 2), "alternate", 8),
                                           ((1, 2, 3, 5), "alternate", 15),
                                           ((2, 3, 4, 2), "alternate", 24),
                                           ((1, 5, 5, 5), "mod5", 100),
                                           ((3, 5, 7, 11), "alternate", 577),
                                           ((1, 8, 8, 80), "mod5", 4096)])
def test_directed_step_streams(fanout, rule, D):
    spec = synth.Spec(name="dirstep", fanout=fanout, role_rule=rule, n_streams=2,
                      requests_per_stream=120, rate_per_s=40.0, len_median=2048.0,
                      len_clip=(16, 16384), n_roots=6, root_blocks=(1024,), n_keys=2000,
                      log2_cap=12, tables="shared", telemetry="shared", cap_tokens=60_000)
    w = synth.make_workload(spec)
    assert w.D == D
    _, x, out = run_gpu(w, cap=spec.cap_tokens, directed=True)
    assert int(out.status.item()) == 0
    near = 0
    for s in range(w.n_streams):
        near += check_stream(w, s, out, cap=spec.cap_tokens, directed=True).near_ties
    assert near <= 3
