"""The allocation-free prefix match agrees with the regular one.

Some callers of this library cannot allocate device memory while they score
requests: a scheduler plugin running inside a serving engine whose memory pool
already owns the GPU, or a request path that must never call cudaMalloc.
netkv_prefix_match_static serves them with a fixed device array compiled into
the library.  This test calls it through the C ABI twice in a row, on two
different workloads, and checks each result against netkv_prefix_match on the
same inputs (bit-exact, the tolerance of every integer output here), then checks
that an oversized call is refused.  It runs alone or after the other tests.
"""
import numpy as np
import pytest

import synth
from synth import stage

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.init()


def _inputs(w):
    from paper_2606_03910_gb300 import netkv
    cap = netkv.index_log2_capacity(synth.distinct_keys_per_group(w))
    index = torch.empty(netkv.netkv_cache_index_bytes(w.n_sets, w.D, cap) // 8, dtype=torch.int64,
                        device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    netkv.netkv_cache_build(index, w.n_sets, w.D, cap, stage.keys(w, 0, w.n_sets),
                            stage.key_offsets(w, w.n_sets * w.D), st)
    ra = stage.request_arrays(w)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return index, cap, stage.chains(w), ra["chain_off"], ra["set_off"]


def _compare(w):
    from paper_2606_03910_gb300 import netkv
    tables, cap, chains, chain_off, set_off = _inputs(w)
    so = set_off if w.n_sets > 1 else None
    ref = torch.full((w.R, w.D), -1, dtype=torch.int16, device="cuda")
    st_ref = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = torch.empty(netkv.netkv_prefix_match_workspace_size(w.R), dtype=torch.uint8, device="cuda")
    netkv.netkv_prefix_match(tables, w.D, cap, w.n_sets, chains, chain_off, w.R, so,
                             ref, st_ref, workspace=ws)
    got = torch.full((w.R, w.D), -1, dtype=torch.int16, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    netkv.netkv_prefix_match_static(tables, w.D, cap, w.n_sets, chains, chain_off,
                                    w.R, so, got, st)
    torch.cuda.synchronize()
    assert int(st.item()) == int(st_ref.item()) == 0
    assert torch.equal(got, ref)
    return got


def test_static_prefix_match_two_calls_and_limit():
    from paper_2606_03910_gb300 import netkv
    # call 1: one stream, 1,000 requests against 8 caches of 200K blocks
    m1 = _compare(synth.make_workload(synth.config0()))
    assert (m1.cpu().numpy().view(np.uint16) > 0).any()
    # call 2: a different shape (two table sets, 16 decodes) right after; the shared
    # scratch still holds call 1's contents
    m2 = _compare(synth.make_workload(synth.tiny_spec(requests_per_stream=60)))
    assert (m2.cpu().numpy().view(np.uint16) > 0).any()
    # more requests than the fixed scratch holds: refused, nothing written
    R = netkv.NETKV_PREFIX_MATCH_STATIC_MAX_R + 1
    M = torch.full((1, 1), 7, dtype=torch.int16, device="cuda")
    off = torch.zeros(R + 1, dtype=torch.int64, device="cuda")
    tab = torch.zeros(2, dtype=torch.int64, device="cuda")
    with pytest.raises(netkv.NetKVError) as e:
        netkv.netkv_prefix_match_static(tab, 1, 1, 1, tab, off, R, None, M, None)
    assert e.value.code == netkv.NETKV_ELIMIT
    torch.cuda.synchronize()
    assert int(M.item()) == 7
