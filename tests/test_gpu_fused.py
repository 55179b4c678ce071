"""The greedy with the level bottlenecks taken from the utilisation rows inside the
base-score pass (netkv_schedule_streams_util) against netkv_oracle_build(UB) followed by
netkv_schedule_streams with a workspace: decisions, best and second scores and final
loads bit for bit on every launch shape (both base-score kernels, the packed and the
staged walks), and a utilisation outside [0, 1) flagged as the oracle build flags it.
The full-size bench workload runs this form (tests/test_gpu_fullsize.py)."""
import numpy as np
import pytest

import synth
from tests.gpu_common import host, run_gpu

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


SHAPES = [((2, 2, 2, 2), "alternate", 8), ((1, 2, 3, 5), "alternate", 15),
          ((2, 3, 4, 2), "alternate", 24), ((1, 5, 5, 5), "mod5", 100),
          ((3, 5, 7, 11), "alternate", 577), ((1, 8, 8, 80), "mod5", 4096)]


@pytest.mark.parametrize("fanout,rule,D", SHAPES)
def test_fused_equals_ub_path(fanout, rule, D):
    spec = synth.Spec(name="fused", fanout=fanout, role_rule=rule, n_streams=3,
                      requests_per_stream=150, rate_per_s=400.0, len_median=2048.0,
                      len_clip=(16, 16384), n_roots=6, root_blocks=(1024,), n_keys=1500,
                      log2_cap=12, tables="shared", telemetry="per_stream", cap_tokens=30_000)
    w = synth.make_workload(spec)
    assert w.D == D
    sc, x, ref = run_gpu(w)              # oracle build, prefix match, greedy with workspace
    assert int(ref.status.item()) == 0
    sc.fuse_level_bottlenecks = True
    assert sc.fused(x)
    out = sc.alloc_outputs(x.n_snap, x.R, x.n_streams)
    sc.step(x, out)
    torch.cuda.synchronize()
    assert int(out.status.item()) == 0
    for f in ("M", "dec", "best", "second", "load_final"):
        assert torch.equal(getattr(out, f), getattr(ref, f)), f


def test_fused_flags_bad_utilisation():
    w = synth.make_workload(synth.tiny_spec())
    sc, x, ref = run_gpu(w)
    sc.fuse_level_bottlenecks = True
    x.util[0, :] = 1.5
    out = sc.alloc_outputs(x.n_snap, x.R, x.n_streams)
    sc.step(x, out)
    torch.cuda.synchronize()
    used = np.unique(w.snap[w.events[(w.events >> 31) == 0] & 0x7FFFFFFF])
    if 0 in used:
        assert int(out.status.item()) & 1  # NETKV_DEV_EDOMAIN


def test_fused_requires_workspace():
    from paper_2606_03910_gb300 import netkv
    w = synth.make_workload(synth.tiny_spec())
    sc, x, ref = run_gpu(w)
    out = sc.alloc_outputs(x.n_snap, x.R, x.n_streams)
    with pytest.raises(netkv.NetKVError):
        netkv.netkv_schedule_streams_util(sc.topo, x.n_streams, x.weights, x.R, x.length,
                                          x.prefill, x.snap, ref.M, x.util, x.n_snap, x.events,
                                          x.event_off, None, out.dec, out.best, out.second,
                                          out.load_final, out.status, workspace=None)
