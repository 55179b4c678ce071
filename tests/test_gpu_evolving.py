"""GPU parity of the greedy with evolving caches (netkv_schedule_streams_evolving: the
LRU-managed decode caches of the simulator of Sec. VI-B) against the oracle's
evolving-cache greedy, on whole streams.

Checked bit for bit: the prefix hits each arrival was scored with, the decisions (a
near-tie, where the GPU's choice scores within 1e-5 of the oracle's best, is replayed and
counted), the final loads, and every decode's final cache, block by block in recency
order (netkv_lru_export).  Scores are checked within 1e-5.  The cases:
  * caches that start full (every dispatch evicts) and caches with room to grow first,
    on pools of 8, 15, 100 and 577 decodes;
  * two calls in a row, the second continuing from the caches and loads the first left,
    equal to one call;
  * no dispatch at all (nothing fits): the hits are those of the static match;
  * two whole streams of the 4,096-replica workload with 200,000-block caches;
  * host-side rejections of invalid configurations.
"""
import numpy as np
import pytest

import synth
from synth import stage
from tests.gpu_common import THETA, host, make_scorer, rel_close

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


def inputs(w, cap=None):
    from paper_2606_03910_gb300.pipeline import StepInputs, weights_tensor
    ra = stage.request_arrays(w)
    cap = w.spec.cap_tokens if cap is None else cap
    return StepInputs(util=stage.util(w), chains=stage.chains(w), chain_off=ra["chain_off"],
                      set_off=ra["set_off"], length=ra["length"], prefill=ra["prefill"],
                      snap=ra["snap"], events=ra["events"], event_off=ra["event_off"],
                      weights=weights_tensor(w.weights, THETA, cap, synth.BYTES_PER_TOKEN_SHARD))


def run_evolving(w, cap_blocks, cap=None):
    """The whole step with evolving caches: level bottlenecks, then hits and greedy in one
    call, from every stream's own key lists (most recently used first)."""
    assert w.n_sets == w.n_streams  # one table set per stream
    sc = make_scorer(w)
    sc.lru_setup(w.n_streams, cap_blocks)
    sc.lru_reset(stage.keys(w, 0, w.n_sets), stage.key_offsets(w, w.n_sets * w.D))
    x = inputs(w, cap)
    out = sc.alloc_outputs(x.n_snap, x.R, x.n_streams)
    sc.step(x, out)
    torch.cuda.synchronize()
    return sc, x, out


def check_streams(w, sc, out, cap_blocks, cap=None, streams=None):
    """Every stream (or the given ones) against the oracle; returns (near-ties, evicting
    decodes, hits that differ from the static match)."""
    from oracle.workload import run_stream_evolving, stream_hits, stream_inputs
    cap = w.spec.cap_tokens if cap is None else cap
    assert int(out.status.item()) == 0
    dec, best, second = host(out.dec), host(out.best), host(out.second)
    M = host(out.M).view(np.uint16)
    keys, lens = sc.lru_export()
    torch.cuda.synchronize()
    keys, lens = host(keys).view(np.uint64), host(lens)
    near = full = moved = 0
    for s in (range(w.n_streams) if streams is None else streams):
        r0, r1 = int(w.req_off[s]), int(w.req_off[s + 1])
        res = run_stream_evolving(w, s, THETA, cap, synth.BYTES_PER_TOKEN_SHARD, cap_blocks,
                                  hint=dec[r0:r1])
        np.testing.assert_array_equal(M[r0:r1], res.M)
        assert res.mismatches == 0, f"stream {s}: {res.mismatches} unexplained decisions"
        np.testing.assert_array_equal(res.dec, dec[r0:r1])
        ev = w.events[w.event_off[s]:w.event_off[s + 1]]
        arr = (ev[(ev >> 31) == 0] & 0x7FFFFFFF).astype(np.int64) - r0
        assert rel_close(best[r0:r1][arr], res.best[arr]).all()
        assert rel_close(second[r0:r1][arr], res.second[arr]).all()
        np.testing.assert_array_equal(host(out.load_final[s]), res.load)
        for d in range(w.D):
            c = s * w.D + d
            np.testing.assert_array_equal(keys[c, :lens[c]], res.caches[d])
            full += int(lens[c] == cap_blocks)
        near += res.near_ties
        moved += int((res.M != stream_hits(w, stream_inputs(w, s))).sum())
    return near, full, moved


def spec_for(fanout, rule, n_keys, **kw):
    base = dict(name="evolving", fanout=fanout, role_rule=rule, n_streams=2,
                requests_per_stream=120, rate_per_s=400.0, len_median=2048.0,
                len_clip=(16, 16384), n_roots=6, root_blocks=(1024,), n_keys=n_keys,
                log2_cap=12, tables="per_stream", telemetry="per_stream", cap_tokens=60_000)
    base.update(kw)
    return synth.Spec(**base)


SHAPES = [((2, 2, 2, 2), "alternate", 8), ((1, 2, 3, 5), "alternate", 15),
          ((1, 5, 5, 5), "mod5", 100), ((3, 5, 7, 11), "alternate", 577)]


@pytest.mark.parametrize("fanout,rule,D", SHAPES)
@pytest.mark.parametrize("n_keys,cap_blocks", [(1500, 1500), (600, 2500)])
def test_evolving_streams_vs_oracle(fanout, rule, D, n_keys, cap_blocks):
    w = synth.make_workload(spec_for(fanout, rule, n_keys))
    assert w.D == D
    sc, x, out = run_evolving(w, cap_blocks)
    near, full, moved = check_streams(w, sc, out, cap_blocks)
    assert near <= 3
    assert moved > 0            # dispatches changed later hits
    if n_keys == cap_blocks:
        assert full > 0         # caches stayed at capacity: dispatches evicted


def test_evolving_two_calls_equal_one():
    """The first half of every stream's events, then the rest from the caches, loads and
    decisions the first call left: the same hits, decisions, scores, loads and caches."""
    netkv = nk()
    w = synth.make_workload(spec_for((2, 2, 2, 2), "alternate", 1500))
    cap_blocks = 1500
    sc, x, out = run_evolving(w, cap_blocks)
    keys1, lens1 = sc.lru_export()
    sc2 = make_scorer(w)
    sc2.lru_setup(w.n_streams, cap_blocks)
    sc2.lru_reset(stage.keys(w, 0, w.n_sets), stage.key_offsets(w, w.n_sets * w.D))
    o2 = sc2.alloc_outputs(x.n_snap, x.R, x.n_streams)
    sc2.oracle_build(x, o2)
    eo = host(x.event_off)
    mid = (eo[:-1] + eo[1:]) // 2
    first = torch.from_numpy(np.stack([eo[:-1], mid], 1).reshape(-1).astype(np.int64)).cuda()
    second = torch.from_numpy(np.stack([mid, eo[1:]], 1).reshape(-1).astype(np.int64)).cuda()
    n = x.n_streams
    per_stream = netkv.netkv_lru_state_bytes(w.D, sc2.lru_cfg)  # caches of one stream
    # one stream per call: its weights, its caches and its half of the events
    for s in range(n):
        for rng in (first, second):
            off = rng[2 * s:2 * s + 2].contiguous()
            ws = x.weights[32 * s:32 * (s + 1)]
            st = sc2.lru_state.view(torch.uint8)[s * per_stream:]
            load_in = o2.load_final[s:s + 1].clone() if rng is second else None
            lf = torch.empty((1, w.D), dtype=torch.int64, device="cuda")
            netkv.netkv_schedule_streams_evolving(
                sc2.topo, 1, ws, x.R, x.length, x.prefill, x.snap, o2.UB, x.n_snap, x.chains,
                x.chain_off, x.events, off, st, sc2.lru_cfg, load_in, o2.dec, o2.best, o2.second,
                o2.M, lf, o2.status)
            o2.load_final[s:s + 1].copy_(lf)
    torch.cuda.synchronize()
    assert int(o2.status.item()) == 0
    for f in ("M", "dec", "best", "second", "load_final"):
        assert torch.equal(getattr(o2, f), getattr(out, f)), f
    keys2, lens2 = sc2.lru_export()
    torch.cuda.synchronize()
    assert torch.equal(lens1, lens2)
    for c in range(lens1.numel()):
        assert torch.equal(keys1[c, :int(lens1[c])], keys2[c, :int(lens2[c])])


def test_evolving_without_dispatch_is_the_static_match():
    """Nothing fits (capacity 0 tokens): every arrival is rejected, no cache changes, and
    every hit equals the static prefix match of the same caches."""
    from tests.gpu_common import run_gpu
    w = synth.make_workload(spec_for((1, 2, 3, 5), "alternate", 1500))
    _, _, ref = run_gpu(w, cap=0)
    sc, x, out = run_evolving(w, 1500, cap=0)
    assert int(out.status.item()) == 0
    assert (host(out.dec) == -1).all()
    assert torch.equal(out.M, ref.M)


def test_evolving_bench_workload_streams():
    """Two whole streams of the 4,096-replica workload (1,000 requests, 8 decodes) with the
    configs' 200,000-block caches, which start full: every dispatch evicts."""
    spec = synth.config1(2)
    w = synth.make_workload(spec)
    sc, x, out = run_evolving(w, 200_000)
    near, full, moved = check_streams(w, sc, out, 200_000)
    assert near <= 3 and full == 2 * w.D and moved > 0


def test_evolving_invalid_configurations():
    netkv = nk()
    w = synth.make_workload(spec_for((2, 2, 2, 2), "alternate", 100))
    sc = make_scorer(w)
    bad = [netkv.LruConfig(0, 17, 17),       # no capacity
           netkv.LruConfig(1000, 16, 17),    # table too small for a 65,535-block chain
           netkv.LruConfig(1000, 17, 16)]    # log too small
    for cfg in bad:
        assert netkv.netkv_lru_state_bytes(4, cfg) == 0
        st = torch.empty(1 << 20, dtype=torch.int64, device="cuda")
        with pytest.raises(netkv.NetKVError):
            netkv.netkv_lru_init(st, 4, cfg, None, None)
    huge = make_scorer(synth.make_workload(spec_for((1, 8, 8, 80), "mod5", 10, n_streams=1,
                                                    requests_per_stream=2)))
    assert huge.D == 4096
    cfg = netkv.lru_config(100)
    x = inputs(synth.make_workload(spec_for((1, 8, 8, 80), "mod5", 10, n_streams=1,
                                            requests_per_stream=2)))
    out = huge.alloc_outputs(x.n_snap, x.R, x.n_streams)
    st = torch.empty(16, dtype=torch.int64, device="cuda")
    with pytest.raises(netkv.NetKVError):   # more than 1,024 decodes
        netkv.netkv_schedule_streams_evolving(
            huge.topo, 1, x.weights, x.R, x.length, x.prefill, x.snap, out.UB, x.n_snap,
            x.chains, x.chain_off, x.events, x.event_off, st, cfg, None, out.dec, out.best,
            out.second, out.M, out.load_final, out.status)
