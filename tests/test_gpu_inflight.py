"""GPU parity of the greedy with self-contention (netkv_schedule_streams_inflight;
Eq. 4's n_inflight, Algorithm 1 lines 5 and 14, Sec. V-C) against the oracle.

* cap 0 is the plain greedy: bit for bit the no-workspace netkv_schedule_streams.
* The worked example of Sec. III-D end to end: one transfer in flight on tier 2 makes
  d1 cost 2.0 s against 0.4 s on d2.
* Whole streams at high arrival rates on four prefill ranks (transfers overlapping),
  every launch shape
  (packed segments of 8 and 16 lanes, one warp, 256- and 1,024-thread CTAs), caps 1,
  2 and 16: decisions exact (near-ties replayed and counted), transfer times exact
  (a transfer time within one microsecond of the oracle's, the same value rounded from
  fp32 instead of double, is adopted and counted), scores within 1e-5, final loads
  exact.
* A stream with more pending completions than its heap holds reports EFULL.
"""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_common import THETA, host, rel_close, run_gpu

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


def run_inflight(sc, x, out, inflight_cap, arrival, workspace=False):
    """workspace: the form with base scores and s_eff / Bbot computed first."""
    netkv = nk()
    R, S, D = x.R, x.n_streams, sc.D
    dev = out.M.device
    o = dict(dec=torch.full((max(R, 1),), -7, dtype=torch.int32, device=dev),
             best=torch.empty(max(R, 1), dtype=torch.float32, device=dev),
             second=torch.empty(max(R, 1), dtype=torch.float32, device=dev),
             xfer=torch.full((max(R, 1),), -7, dtype=torch.int32, device=dev),
             load=torch.empty((S, D), dtype=torch.int64, device=dev),
             status=torch.zeros(1, dtype=torch.int32, device=dev))
    netkv.netkv_schedule_streams_inflight(sc.topo, S, x.weights, R, x.length, x.prefill, x.snap,
                                          arrival, out.M, out.UB, x.n_snap, x.events, x.event_off,
                                          inflight_cap, x.load_init, o["dec"], o["best"],
                                          o["second"], o["xfer"], o["load"], o["status"],
                                          workspace=torch.empty(
                                              netkv.netkv_schedule_inflight_workspace_size(R, D),
                                              dtype=torch.uint8, device=dev) if workspace else None)
    torch.cuda.synchronize()
    return o


def _workload(spec, n_prefills=None):
    """n_prefills: fold the requests onto that many prefill ranks (contention is per
    prefill, so large pools need it to see transfers in flight)."""
    w = synth.make_workload(spec)
    if n_prefills:
        w.prefill[:] = w.prefill % n_prefills
    sc, x, out = run_gpu(w, cap=spec.cap_tokens)
    arrival = torch.from_numpy(w.arrival_us.astype(np.int64)).cuda()
    return w, sc, x, out, arrival


SHAPES = [((2, 2, 2, 2), "alternate", 8),     # packed: 4 streams a warp, 8 lanes each
          ((1, 2, 3, 5), "alternate", 15),    # packed: 2 streams a warp, 16 lanes each
          ((2, 3, 4, 2), "alternate", 24),    # one warp per stream
          ((1, 5, 5, 5), "mod5", 100),        # 256-thread CTA, one decode each
          ((3, 5, 7, 11), "alternate", 577),  # 256-thread CTA, four each, ragged
          ((1, 8, 8, 80), "mod5", 4096)]      # 1,024-thread CTA, four each


def _spec(fanout, rule, rate=2000.0, rps=120, n_streams=2):
    return synth.Spec(name="inflight", fanout=fanout, role_rule=rule, n_streams=n_streams,
                      requests_per_stream=rps, rate_per_s=rate, len_median=2048.0,
                      len_clip=(16, 16384), n_roots=6, root_blocks=(1024,), n_keys=2000,
                      log2_cap=12, tables="shared", telemetry="shared", cap_tokens=200_000)


@pytest.mark.parametrize("fanout,rule,D", SHAPES)
@pytest.mark.parametrize("ws", [False, True])
def test_inflight_cap0_is_the_plain_greedy(fanout, rule, D, ws):
    """Without workspaces and with them, on each side."""
    netkv = nk()
    w, sc, x, out, arrival = _workload(_spec(fanout, rule))
    assert w.D == D
    o = run_inflight(sc, x, out, 0, arrival, workspace=ws)
    assert int(o["status"].item()) == 0
    plain = sc.alloc_outputs(x.n_snap, x.R, x.n_streams)
    netkv.netkv_schedule_streams(sc.topo, x.n_streams, x.weights, x.R, x.length, x.prefill,
                                 x.snap, out.M, out.UB, x.n_snap, x.events, x.event_off,
                                 x.load_init, plain.dec, plain.best, plain.second,
                                 plain.load_final, plain.status,
                                 workspace=torch.empty(netkv.netkv_schedule_workspace_size(x.R, D),
                                                       dtype=torch.uint8, device="cuda")
                                 if ws else None)
    torch.cuda.synchronize()
    assert torch.equal(o["dec"], plain.dec)
    assert torch.equal(o["best"], plain.best) and torch.equal(o["second"], plain.second)
    assert torch.equal(o["load"], plain.load_final)
    assert torch.equal(o["xfer"] >= 0, plain.dec >= 0)


@pytest.mark.parametrize("fanout,rule,D", SHAPES)
@pytest.mark.parametrize("icap,ws", [(1, False), (2, False), (16, False), (2, True), (16, True)])
def test_inflight_streams_vs_oracle(fanout, rule, D, icap, ws):
    from oracle.workload import run_stream_inflight
    w, sc, x, out, arrival = _workload(_spec(fanout, rule), n_prefills=4)
    o = run_inflight(sc, x, out, icap, arrival, workspace=ws)
    assert int(o["status"].item()) == 0
    dec, best, second = host(o["dec"]), host(o["best"]), host(o["second"])
    xfer, load = host(o["xfer"]), host(o["load"])
    M = host(out.M).view(np.uint16)
    changed = adopted = near = 0
    for s in range(w.n_streams):
        r0, r1 = int(w.req_off[s]), int(w.req_off[s + 1])
        res = run_stream_inflight(w, s, THETA, w.spec.cap_tokens, synth.BYTES_PER_TOKEN_SHARD,
                                  icap, hint=dec[r0:r1], xfer_hint=xfer[r0:r1])
        np.testing.assert_array_equal(M[r0:r1], res.M)
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
        plain = run_stream_inflight(w, s, THETA, w.spec.cap_tokens, synth.BYTES_PER_TOKEN_SHARD, 0,
                                    M=res.M)
        changed += int((plain.dec != res.dec).sum() + (plain.best[arr] != res.best[arr]).sum())
    assert near <= 3 and adopted <= 3
    assert changed > 0       # transfers overlap: contention changed scores or decisions


def test_inflight_worked_example_on_gpu():
    """Sec. III-D through the library: request A (no hits) to d1, in flight for 2 s;
    request B at 1 ms sees T_d1 = 2.0 s (one in flight on tier 2) and T_d2 = 0.4 s."""
    netkv = nk()
    from paper_2606_03910_gb300.pipeline import weights_tensor
    fanout = (2, 2, 2, 2)
    role = np.zeros(16, np.uint8)
    role[[4, 8]] = 1
    L = oracle.used_links(fanout)
    topo = netkv.netkv_topology_create(fanout, role, (100e9, 50e9, 6.25e9, 3.125e9),
                                       (0.0, 0.0, 0.0, 0.0), L)
    u = torch.full((1, L), 0.2, dtype=torch.float32, device="cuda")
    N = 16
    UB = torch.empty((1, N, 4), dtype=torch.float32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    netkv.netkv_oracle_build(topo, u, 1, 1.0, None, UB, st)
    R = 2
    i32 = lambda a: torch.tensor(a, dtype=torch.int32, device="cuda")
    length = i32([100_000, 100_000])
    zeros = i32([0, 0])
    arrival = torch.tensor([0, 1000], dtype=torch.int64, device="cuda")
    M = torch.tensor([[0, 0], [3125, 5625]], dtype=torch.int16, device="cuda")
    events = torch.tensor([0, 1, 0x80000000, 0x80000001], dtype=torch.int64).to(torch.int32).cuda()
    event_off = torch.tensor([0, 4], dtype=torch.int64, device="cuda")
    wts = weights_tensor(np.array([[1.0, 0.0, 0.0]], np.float32), 0.0, 10 ** 7, 100_000, device="cuda")
    dec = torch.full((R,), -7, dtype=torch.int32, device="cuda")
    best = torch.empty(R, dtype=torch.float32, device="cuda")
    second = torch.empty(R, dtype=torch.float32, device="cuda")
    xfer = torch.empty(R, dtype=torch.int32, device="cuda")
    lf = torch.empty((1, 2), dtype=torch.int64, device="cuda")
    netkv.netkv_schedule_streams_inflight(topo, 1, wts, R, length, zeros, zeros, arrival, M, UB, 1,
                                          events, event_off, 16, None, dec, best, second, xfer,
                                          lf, st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert host(dec).tolist() == [0, 1]
    assert host(xfer).tolist() == [2_000_000, 400_000]
    assert float(best[1]) == pytest.approx(0.4, rel=1e-6)
    assert float(second[1]) == pytest.approx(2.0, rel=1e-6)
    assert host(lf).tolist() == [[0, 0]]


def test_inflight_heap_overflow_reported():
    """800 arrivals a microsecond apart with millisecond transfers: more pending
    completions than a packed stream's 256-entry heap; the call flags EFULL."""
    netkv = nk()
    spec = synth.tiny_spec(n_streams=1, requests_per_stream=800, rate_per_s=1e6,
                           cap_tokens=10 ** 9)
    w, sc, x, out, arrival = _workload(spec)
    o = run_inflight(sc, x, out, 16, arrival)
    assert int(o["status"].item()) & netkv.NETKV_DEV_EFULL
