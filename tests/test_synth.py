"""Determinism and shape checks of the synthetic input generators (no GPU)."""
import numpy as np

import synth


def test_deterministic_and_seeded():
    a = synth.make_workload(synth.tiny_spec())
    b = synth.make_workload(synth.tiny_spec())
    np.testing.assert_array_equal(a.chains(), b.chains())
    np.testing.assert_array_equal(a.events, b.events)
    c = synth.make_workload(synth.tiny_spec(seed0=7))
    assert not np.array_equal(a.length, c.length)


def test_events_are_ordered_and_complete():
    w = synth.make_workload(synth.config0())
    ev = w.events
    r = ev & 0x7FFFFFFF
    dep = ev >> 31
    t = np.where(dep == 1, w.depart_us[r], w.arrival_us[r])
    assert (np.diff(t) >= 0).all()
    assert np.bincount(r[dep == 0], minlength=w.R).tolist() == [1] * w.R
    assert np.bincount(r[dep == 1], minlength=w.R).tolist() == [1] * w.R
    first = {}
    for i, (rr, dd) in enumerate(zip(r, dep)):
        if dd == 0:
            first[rr] = i
        else:
            assert first[rr] < i


def test_config_shapes():
    w = synth.make_workload(synth.config0())
    assert (w.P, w.D, w.L, w.R) == (8, 8, 44, 1000)
    assert (w.keys(0, 3) != 0).all() and len(w.keys(0, 3)) == 200_000
    u = w.util(0, 10)
    assert u.dtype == np.float32 and (u >= 0).all() and (u < 0.9).all()
    assert synth.used_links(synth.config3()) == 21_920
    assert synth.used_links(synth.config2()) == 10_960
    assert synth.used_links(synth.config4()) == 2_740
    assert synth.config4_root_blocks()[0] == 256 and synth.config4_root_blocks()[-1] == 7680
    assert synth.CAP_TOKENS == 549_316
    s3 = synth.config3(n_snapshots=2)
    w3 = synth.make_workload(s3)
    assert (w3.P, w3.D, w3.L) == (2048, 8192, 24_576)
    u3 = w3.util()
    hot = synth.hot_links(s3, 0)
    assert len(hot) == 1096 and (u3[:, hot] >= 0.85).all() and (u3 < 1).all()


def test_grid_weights():
    w = synth.stream_weights(synth.config1(), 4096)
    assert w.shape == (4096, 3)
    assert len({tuple(x) for x in w}) == 4096
