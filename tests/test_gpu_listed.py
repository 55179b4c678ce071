"""The listed walk of pools of 1,025 .. 4,096 decodes against the staged walk, bit for bit.

With a workspace of netkv_schedule_workspace_size(R, D) bytes the base-score pass also
writes each arrival's candidate list (the pool's 32 smallest base scores) and bound, and the
greedy rescans only arrivals the bound does not certify; a workspace holding only the
base-score rows (R * D * 4 bytes) runs the staged walk over every candidate.  Both are the exact argmin of Algorithm 1 on the same
fp32 scores, so decisions, best and second scores and final loads must agree exactly, on
workloads that certify almost every arrival and on ones built to defeat the bounds: a load
weight that dominates the score, a tight capacity, initial loads (negative ones too), zero
and negative load weights, and pools of 2 to 4 chunks of 1,024 decodes, ragged ones too.  Oracle parity of the
listed walk is covered where the bench shapes run (tests/test_gpu_parity.py,
tests/test_gpu_fused.py, tests/test_gpu_configs.py)."""
import numpy as np
import pytest

import synth
from tests.gpu_common import THETA, run_gpu

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


SHAPES = [((1, 7, 11, 17), 1047),   # two chunks, the second of 23 decodes; D % 4 != 0
          ((1, 8, 8, 40), 2048),
          ((1, 7, 11, 49), 3018),   # ragged: scalar row reads in the full scans
          ((1, 8, 8, 80), 4096)]


def _workload(fanout, n_streams=3, requests=400, cap=60_000):
    spec = synth.Spec(name="listed", fanout=fanout, role_rule="mod5", n_streams=n_streams,
                      requests_per_stream=requests, rate_per_s=60.0, len_median=2048.0,
                      len_clip=(16, 16384), n_roots=6, root_blocks=(1024,), n_keys=2000,
                      log2_cap=12, tables="shared", telemetry="shared", cap_tokens=cap)
    w = synth.make_workload(spec)
    sc, x, out = run_gpu(w, cap=cap)
    assert int(out.status.item()) == 0
    return w, sc, x, out


def _weights(w, scale_load=1.0, cap=60_000, w_load=None):
    from paper_2606_03910_gb300.pipeline import weights_tensor
    wt = w.weights.copy()
    wt[:, 2] *= np.float32(scale_load)
    if w_load is not None:
        wt[:, 2] = np.float32(w_load)
    return weights_tensor(wt, THETA, cap, synth.BYTES_PER_TOKEN_SHARD)


def _run(sc, x, out, weights, load_init, ws_bytes, util=False):
    netkv = nk()
    o = sc.alloc_outputs(x.n_snap, x.R, x.n_streams)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
    if util:
        netkv.netkv_schedule_streams_util(sc.topo, x.n_streams, weights, x.R, x.length,
                                          x.prefill, x.snap, out.M, x.util, x.n_snap, x.events,
                                          x.event_off, load_init, o.dec, o.best, o.second,
                                          o.load_final, o.status, workspace=ws)
    else:
        netkv.netkv_schedule_streams(sc.topo, x.n_streams, weights, x.R, x.length, x.prefill,
                                     x.snap, out.M, out.UB, x.n_snap, x.events, x.event_off,
                                     load_init, o.dec, o.best, o.second, o.load_final,
                                     o.status, workspace=ws)
    torch.cuda.synchronize()
    return o


def _assert_same(a, b):
    assert int(a.status.item()) == int(b.status.item())
    for f in ("dec", "best", "second", "load_final"):
        assert torch.equal(getattr(a, f), getattr(b, f)), f


def _sizes(R, D):
    netkv = nk()
    full = netkv.netkv_schedule_workspace_size(R, D)
    rows = (R * D * 4 + 255) // 256 * 256
    assert full > rows  # the lists need room beyond the rows
    return full, rows


@pytest.mark.parametrize("fanout,D", SHAPES)
@pytest.mark.parametrize("util", [False, True])
def test_listed_equals_staged(fanout, D, util):
    w, sc, x, out = _workload(fanout)
    assert w.D == D
    full, rows = _sizes(x.R, D)
    wt = _weights(w)
    a = _run(sc, x, out, wt, None, full, util)
    b = _run(sc, x, out, wt, None, rows, util)
    assert int(a.status.item()) == 0
    _assert_same(a, b)
    assert (a.dec.cpu().numpy() >= 0).sum() > 0


@pytest.mark.parametrize("fanout,D", [SHAPES[0], SHAPES[3]])
@pytest.mark.parametrize("case", ["load_heavy", "tight_cap", "load_init", "negative_init",
                                  "zero_load_weight", "negative_load_weight"])
def test_listed_against_the_bounds(fanout, D, case):
    cap = 60_000
    w, sc, x, out = _workload(fanout, cap=cap)
    full, rows = _sizes(x.R, D)
    rng = np.random.default_rng(7)
    load_init = None
    wt = _weights(w, cap=cap)
    if case == "load_heavy":      # the load term outweighs the base scores: few certify
        wt = _weights(w, scale_load=1e4, cap=cap)
    elif case == "tight_cap":     # most candidates infeasible
        wt = _weights(w, cap=4_000)
    elif case == "load_init":     # no idle decode: the bound's load floor is positive
        load_init = torch.from_numpy(rng.integers(1, 20_000, (x.n_streams, D)).astype(np.int64)).cuda()
    elif case == "negative_init":  # a negative load turns the tie rule off
        li = rng.integers(0, 20_000, (x.n_streams, D)).astype(np.int64)
        li[:, 5] = -3
        load_init = torch.from_numpy(li).cuda()
    elif case == "zero_load_weight":
        wt = _weights(w, cap=cap, w_load=0.0)
    elif case == "negative_load_weight":  # bounds do not hold: every arrival is scanned
        wt = _weights(w, cap=cap, w_load=-0.5)
    a = _run(sc, x, out, wt, load_init, full)
    b = _run(sc, x, out, wt, load_init, rows)
    _assert_same(a, b)


def test_workspace_size_grows_only_for_listed_pools():
    netkv = nk()
    for D in (8, 32, 256, 1024):
        assert netkv.netkv_schedule_workspace_size(1000, D) == (1000 * D * 4 + 255) // 256 * 256
    r256 = lambda b: (b + 255) // 256 * 256
    for D in (1025, 4096):
        nc = (D + 1023) // 1024  # chunk lists of the base pass, then the pool's merged list
        lists = r256(1000 * nc * 32 * 8) + r256(1000 * nc * 8) + r256(1000 * 32 * 8) + r256(1000 * 8)
        assert netkv.netkv_schedule_workspace_size(1000, D) == (1000 * D * 4 + 255) // 256 * 256 + lists
