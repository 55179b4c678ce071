"""Helpers shared by the GPU parity tests: run the CUDA path on a generated
workload through the C ABI, run the oracle on the same generated inputs, and
compare element by element."""
from __future__ import annotations

import numpy as np

import synth
from synth import stage

THETA = float(np.float32(synth.THETA_S_PER_TOKEN))
REL = 1e-5


def rel_close(a, b, rel=REL):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    both_inf = np.isinf(a) & np.isinf(b) & (np.sign(a) == np.sign(b))
    ok = both_inf | (np.abs(a - b) <= rel * np.maximum(np.abs(a), np.abs(b)))
    return ok


def index_log2(w):
    from paper_2606_03910_gb300 import netkv
    return netkv.index_log2_capacity(synth.distinct_keys_per_group(w))


def make_scorer(w, device="cuda"):
    from paper_2606_03910_gb300.pipeline import Scorer
    spec = w.spec
    return Scorer(spec.fanout, w.role, spec.tier_bw, spec.tier_lat, w.L, w.n_sets,
                  index_log2(w), device=device)


def run_gpu(w, sc=None, cap=None, load_init=None, directed=False, tiers=False):
    """Whole path on the GPU for workload w; returns (scorer, inputs, outputs).
    directed: links carry the generator's upward and downward utilisation rows."""
    import torch
    from paper_2606_03910_gb300.pipeline import StepInputs, weights_tensor
    sc = sc or make_scorer(w)
    keys = stage.keys(w, 0, w.n_sets)
    sc.load_caches(keys, stage.key_offsets(w, w.n_sets * w.D))
    ra = stage.request_arrays(w)
    cap = w.spec.cap_tokens if cap is None else cap
    if tiers:
        sc.oracle_mode = "tiers"
    x = StepInputs(util=stage.util(w, direction="tiers" if tiers else "up"),
                   chains=stage.chains(w), chain_off=ra["chain_off"],
                   set_off=ra["set_off"], length=ra["length"], prefill=ra["prefill"],
                   snap=ra["snap"], events=ra["events"], event_off=ra["event_off"],
                   weights=weights_tensor(w.weights, THETA, cap, synth.BYTES_PER_TOKEN_SHARD),
                   load_init=load_init,
                   util_down=stage.util(w, direction="down") if directed else None)
    out = sc.alloc_outputs(x.n_snap, x.R, x.n_streams)
    sc.step(x, out)
    torch.cuda.synchronize()
    return sc, x, out


def host(t):
    return t.detach().cpu().numpy()


def check_stream(w, s, out, cap=None, M_gpu=None, M_expect=None, directed=False, tiers=False):
    """Oracle on stream s with the GPU decisions as near-tie hints; asserts parity.
    M_expect: the stream's prefix hits for the oracle's greedy where its own per-stream
    cache sets would not fit (the generator's constructed hits).  Returns the oracle result."""
    from oracle.workload import run_stream
    cap = w.spec.cap_tokens if cap is None else cap
    import torch
    r0, r1 = int(w.req_off[s]), int(w.req_off[s + 1])
    dec = host(out.dec[r0:r1])
    res = run_stream(w, s, THETA, cap, synth.BYTES_PER_TOKEN_SHARD, hint=dec, M=M_expect,
                     directed=directed, tiers=tiers)
    # prefix hits: bit-exact
    if M_gpu is None:
        M_gpu = host(out.M[r0:r1]).view(np.uint16)
    np.testing.assert_array_equal(M_gpu, res.M)
    # decisions: exact except near-ties (counted), no unexplained mismatch
    assert res.mismatches == 0, f"stream {s}: {res.mismatches} unexplained decision mismatches"
    np.testing.assert_array_equal(res.dec, dec)
    # scores of every arrival within 1e-5 relative
    arrivals = w.events[w.event_off[s]:w.event_off[s + 1]]
    arr = (arrivals[(arrivals >> 31) == 0] & 0x7FFFFFFF).astype(np.int64) - r0
    gb = host(out.best[r0:r1])[arr]
    gs = host(out.second[r0:r1])[arr]
    assert rel_close(gb, res.best[arr]).all(), "best scores differ"
    assert rel_close(gs, res.second[arr]).all(), "second-best scores differ"
    np.testing.assert_array_equal(host(out.load_final[s]), res.load)
    # level bottlenecks of the snapshots this stream read
    UB = host(out.UB[torch.from_numpy(res.snaps).to(out.UB.device)])
    assert rel_close(UB, res.UB).all(), "level bottlenecks differ"
    return res
