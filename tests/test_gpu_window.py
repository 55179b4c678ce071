"""The windowed walk of pools of at most 16 decodes against another kernel, bit for bit.

With a workspace, pools of up to 16 decodes run the windowed walk: events in windows of 32,
each departure's decode found through small per-window tables keyed by the request index
(mod 64), released tokens pre-summed per arrival and decode.  Self-contention at counter cap 0
with its workspace is the same greedy (Algorithm 1 on the same fp32 base scores and load
term) computed by the packed per-event walk, so decisions, best and second scores, final
loads and the status word must be equal.  The event lists here are built to reach every
branch of the window: request indices renumbered at random (arrivals of neighbouring windows
collide in the tables), departures right after their arrival (same window, next window, or
later), requests that never depart, lengths of 2^27 tokens and more (released one by one),
zero-length arrivals, out-of-range prefill ranks and request indices (flagged), initial
loads, and stream counts that leave segments of a warp empty.  Renumbering the requests
must not change any result.  Oracle parity of the windowed walk on generated streams is in
tests/test_gpu_parity.py, tests/test_gpu_fused.py and tests/test_gpu_fullsize.py."""
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


SHAPES = [((1, 1, 2, 3), 3, 5),     # 8-lane segments, 5 of 8 lanes idle; 5 streams
          ((2, 2, 2, 2), 8, 7),     # 8-lane segments, 4 streams a warp; 7 streams
          ((1, 2, 3, 5), 15, 5),    # 16-lane segments, 2 streams a warp; D % 4 != 0
          ((2, 2, 2, 4), 16, 3)]    # 16-lane segments, 16-byte row copies


def _events(rng, r0, r1, gaps):
    """Arrivals of requests r0..r1-1 in order; request i departs after gaps[i] more arrivals
    (a negative gap: it never departs)."""
    out, pending = [], []          # pending: [events left, r]
    for r in range(r0, r1):
        out.append(r)
        for p in pending:
            p[0] -= 1
        due = [p for p in pending if p[0] <= 0]
        pending = [p for p in pending if p[0] > 0]
        for _, rr in sorted(due, key=lambda p: p[1]):
            out.append(rr | 0x80000000)
        g = int(gaps[r - r0])
        if g == 0:
            out.append(r | 0x80000000)
        elif g > 0:
            pending.append([g, r])
    for _, rr in sorted(pending):
        out.append(rr | 0x80000000)
    return out


def _case(fanout, n_streams, rps=300, seed=0, huge=False, bad=False):
    """Generated requests with hand-built event lists; returns everything both walks need,
    in the original numbering and renumbered at random."""
    spec = synth.Spec(name="window", fanout=fanout, role_rule="alternate", n_streams=n_streams,
                      requests_per_stream=rps, rate_per_s=400.0, len_median=2048.0,
                      len_clip=(16, 16384), n_roots=6, root_blocks=(1024,), n_keys=2000,
                      log2_cap=12, tables="shared", telemetry="shared", cap_tokens=60_000)
    w = synth.make_workload(spec)
    sc, x, out = run_gpu(w)
    assert int(out.status.item()) == 0
    rng = np.random.default_rng(seed)
    R = w.R
    length = w.length.astype(np.int64).copy()
    prefill = w.prefill.astype(np.int64).copy()
    snap = host32(x.snap)
    if huge:   # released one by one: above 2^27 tokens a window's sum could overflow 32 bits
        length[rng.choice(R, size=max(1, R // 20), replace=False)] = (1 << 27) + 12345
    if bad:
        length[rng.choice(R, size=3, replace=False)] = 0          # EDOMAIN
        prefill[rng.choice(R, size=3, replace=False)] = sc.P      # ERANGE
    ev, off = [], [0]
    for s in range(n_streams):
        r0, r1 = int(w.req_off[s]), int(w.req_off[s + 1])
        gaps = rng.choice([-1, 0, 1, 2, 3, 5, 8, 13, 20, 31, 32, 33, 40, 64, 200],
                          size=r1 - r0)
        e = _events(rng, r0, r1, gaps)
        if bad and s == 0:
            e.insert(len(e) // 2, R + 5)                     # out-of-range arrival: ERANGE
            e.insert(len(e) // 3, (R + 7) | 0x80000000)      # out-of-range departure: ERANGE
        ev += e
        off.append(len(ev))
    ev = np.array(ev, dtype=np.uint32)
    perm = rng.permutation(R).astype(np.int64)   # request r becomes perm[r]
    return dict(w=w, sc=sc, x=x, out=out, length=length, prefill=prefill, snap=snap,
                arrival_us=w.arrival_us.astype(np.int64), events=ev,
                event_off=np.array(off, dtype=np.int64), perm=perm, M=out.M,
                cap=(1 << 40) if huge else 60_000)


def host32(t):
    return t.detach().cpu().numpy().astype(np.int64)


def _renumber(c):
    perm = c["perm"]
    R = len(perm)
    inv = np.argsort(perm)                       # new index -> old index
    ev = c["events"].astype(np.int64)
    r = ev & 0x7FFFFFFF
    ok = r < R
    r2 = np.where(ok, perm[np.minimum(r, R - 1)], r)
    ev2 = ((ev & 0x80000000) | r2).astype(np.uint32)
    M2 = c["M"][torch.from_numpy(inv).to(c["M"].device)]
    return dict(length=c["length"][inv], prefill=c["prefill"][inv], snap=c["snap"][inv],
                arrival_us=c["arrival_us"][inv], events=ev2, M=M2)


def _run(c, arrays, walk, load_init=None):
    netkv = nk()
    sc, x, out = c["sc"], c["x"], c["out"]
    dev = "cuda"
    R, S, D = x.R, x.n_streams, sc.D
    t32 = lambda a: torch.from_numpy(np.asarray(a).astype(np.uint32).view(np.int32)).to(dev)
    length, prefill, snap = t32(arrays["length"]), t32(arrays["prefill"]), t32(arrays["snap"])
    events = t32(arrays["events"])
    event_off = torch.from_numpy(c["event_off"]).to(dev)
    from paper_2606_03910_gb300.pipeline import weights_tensor
    wt = weights_tensor(c["w"].weights, THETA, c["cap"], synth.BYTES_PER_TOKEN_SHARD)
    o = dict(dec=torch.full((R,), -1, dtype=torch.int32, device=dev),
             best=torch.full((R,), 7.0, dtype=torch.float32, device=dev),
             second=torch.full((R,), 7.0, dtype=torch.float32, device=dev),
             load=torch.empty((S, D), dtype=torch.int64, device=dev),
             status=torch.zeros(1, dtype=torch.int32, device=dev))
    if walk == "window":
        ws = torch.empty(netkv.netkv_schedule_workspace_size(R, D), dtype=torch.uint8, device=dev)
        netkv.netkv_schedule_streams(sc.topo, S, wt, R, length, prefill, snap, arrays["M"],
                                     out.UB, x.n_snap, events, event_off, load_init, o["dec"],
                                     o["best"], o["second"], o["load"], o["status"],
                                     workspace=ws)
    else:   # self-contention at cap 0 with its workspace: the packed per-event walk
        ws = torch.empty(netkv.netkv_schedule_inflight_workspace_size(R, D), dtype=torch.uint8,
                         device=dev)
        xfer = torch.empty(R, dtype=torch.int32, device=dev)
        # arrival times in event order, so that the completion heap drains (a transfer
        # still pending past the heap's 256 entries would only set EFULL)
        arrival = torch.from_numpy(arrays["arrival_us"]).to(dev)
        netkv.netkv_schedule_streams_inflight(sc.topo, S, wt, R, length, prefill, snap, arrival,
                                              arrays["M"], out.UB, x.n_snap, events, event_off,
                                              0, load_init, o["dec"], o["best"], o["second"],
                                              xfer, o["load"], o["status"], workspace=ws)
    torch.cuda.synchronize()
    return o


def _assert_same(a, b):
    for f in ("status", "dec", "best", "second", "load"):
        assert torch.equal(a[f], b[f]), f


@pytest.mark.parametrize("fanout,D,n_streams", SHAPES)
@pytest.mark.parametrize("kind", ["plain", "huge", "bad", "load_init"])
def test_window_equals_packed_walk(fanout, D, n_streams, kind):
    c = _case(fanout, n_streams, huge=kind == "huge", bad=kind == "bad")
    assert c["sc"].D == D
    load_init = None
    if kind == "load_init":
        rng = np.random.default_rng(3)
        li = rng.integers(-50, 30_000, (n_streams, D)).astype(np.int64)
        load_init = torch.from_numpy(li).cuda()
    orig = dict(length=c["length"], prefill=c["prefill"], snap=c["snap"],
                arrival_us=c["arrival_us"], events=c["events"], M=c["M"])
    ren = _renumber(c)
    for arrays in (orig, ren):
        a = _run(c, arrays, "window", load_init)
        b = _run(c, arrays, "packed", load_init)
        _assert_same(a, b)
        st = int(a["status"].item())
        if kind == "bad":
            assert st == (nk().NETKV_DEV_EDOMAIN | nk().NETKV_DEV_ERANGE)
        else:
            assert st == 0
        assert (a["dec"] >= 0).sum().item() > 0
    # renumbering the requests changes no result
    a = _run(c, orig, "window", load_init)
    b = _run(c, ren, "window", load_init)
    perm = torch.from_numpy(c["perm"]).cuda()
    for f in ("dec", "best", "second"):
        assert torch.equal(a[f], b[f][perm]), f
    assert torch.equal(a["load"], b["load"])
