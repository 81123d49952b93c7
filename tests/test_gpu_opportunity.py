"""The opportunity grid on the GPU (rc_opportunity_grid: F, P*, U for every
(deadline, threshold) pair, one GPU thread per route and pair) against the
oracle on small sets and against the library's host counts (themselves
checked against the oracle in test_opportunity) on the replay, under the
paper's three groupings (Section 5.2)."""
import numpy as np
import pytest

import oracle
import rc_workload as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rc():
    import paper_2608_12123_gb300 as m
    return m


@pytest.mark.parametrize("seed", range(5))
def test_small_sets_every_pair_against_the_oracle(rc, seed):
    rng = np.random.default_rng(100 + seed)
    for _ in range(12):
        n = int(rng.integers(0, 90))
        R = int(rng.integers(1, 5))
        t = rng.integers(-30, 150, n).astype(np.int64)
        r = rng.integers(0, R, n).astype(np.uint32)
        ks = [1, 2, 3, 7]
        ds = [1, 4, 13, 40]
        origin = int(rng.integers(-5, 5))
        got = rc.rc_opportunity_grid(t, r, R, ks, ds, origin)
        for a, d in enumerate(ds):
            for b, k in enumerate(ks):
                want = (oracle.fixed_count(t, r, R, k, d, origin), oracle.exact_count(t, r, R, k, d),
                        oracle.upper_count(t, r, R, k, d))
                assert tuple(int(v) for v in got[a, b]) == want, (n, R, d, k)


@pytest.mark.parametrize("grouping", ["route", "class", "pooled"])
def test_replay_grid_against_host_counts(rc, grouping):
    panel = wl.make_panel()
    a = wl.make_arrivals(10_000, panel)
    if grouping == "route":
        route, R = a.route, panel.n_labels
    elif grouping == "class":
        route, R = (a.route % 8).astype(np.uint32), 8
    else:
        route, R = np.zeros(a.n, np.uint32), 1
    ks = [32, 64, 128, 256]
    ds = [10_000_000, 25_000_000, 50_000_000, 100_000_000, 250_000_000]
    got = rc.rc_opportunity_grid(a.t_ns, route, R, ks, ds, 0)
    for i, d in enumerate(ds):
        for j, k in enumerate(ks):
            c = rc.rc_opportunity(a.t_ns, route, R, k, d, 0)
            assert tuple(int(v) for v in got[i, j]) == (c["fixed"], c["exact"], c["upper"]), (d, k)
            assert c["fixed"] <= c["exact"] <= c["upper"]


def test_empty_set_and_bad_arguments(rc):
    z = rc.rc_opportunity_grid(np.zeros(0, np.int64), np.zeros(0, np.uint32), 1, [4], [5], 0)
    assert z.shape == (1, 1, 3) and not z.any()
    with pytest.raises(rc.RcError):
        rc.rc_opportunity_grid(np.array([1], np.int64), np.array([0], np.uint32), 1, [0], [5], 0)
    with pytest.raises(rc.RcError):
        rc.rc_opportunity_grid(np.array([1], np.int64), np.array([2], np.uint32), 2, [1], [5], 0)
    with pytest.raises(rc.RcError):  # at most 32 thresholds per call
        rc.rc_opportunity_grid(np.array([1], np.int64), np.array([0], np.uint32), 1, list(range(1, 34)), [5], 0)


def test_events_out_of_time_order(rc):
    rng = np.random.default_rng(7)
    t = rng.integers(0, 500, 300).astype(np.int64)
    r = rng.integers(0, 3, 300).astype(np.uint32)
    perm = rng.permutation(300)
    a = rc.rc_opportunity_grid(t, r, 3, [2, 5], [10, 40], 0)
    b = rc.rc_opportunity_grid(t[perm], r[perm], 3, [2, 5], [10, 40], 0)
    c = rc.rc_opportunity_grid(np.sort(t), r[np.argsort(t, kind="stable")], 3, [2, 5], [10, 40], 0)
    assert np.array_equal(a, b) and np.array_equal(a, c)
