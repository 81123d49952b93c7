"""The library's opportunity counts (rc_opportunity: F of Eq. 2, P* of Eq. 6 /
Algorithm 1, U of Eqs. 3-4) against the oracle's, which is pinned by brute
force and closed forms in test_oracle_packing.  Host code only: no GPU."""
import numpy as np
import pytest

import oracle
import rc_workload as wl


@pytest.fixture(scope="module")
def rc():
    import paper_2608_12123_gb300 as m
    return m


def _want(t, r, R, K, d, origin=0):
    return dict(fixed=oracle.fixed_count(t, r, R, K, d, origin), exact=oracle.exact_count(t, r, R, K, d),
                upper=oracle.upper_count(t, r, R, K, d))


@pytest.mark.parametrize("seed", range(6))
def test_random_small_sets_any_input_order(rc, seed):
    rng = np.random.default_rng(seed)
    for _ in range(60):
        n = int(rng.integers(0, 80))
        R = int(rng.integers(1, 5))
        K = int(rng.integers(1, 7))
        d = int(rng.integers(1, 25))
        t = rng.integers(-40, 120, n).astype(np.int64)  # ties and times before the origin
        r = rng.integers(0, R, n).astype(np.uint32)
        origin = int(rng.integers(-10, 10))
        got = rc.rc_opportunity(t, r, R, K, d, origin)
        want = _want(t, r, R, K, d, origin)
        assert (got["fixed"], got["exact"], got["upper"]) == (want["fixed"], want["exact"], want["upper"])
        assert got["n"] == n
        assert got["fixed"] <= got["exact"] <= got["upper"] <= n  # Proposition 1


def test_replay_workload_matches_oracle(rc):
    panel = wl.make_panel()
    a = wl.make_arrivals(10_000, panel)
    for K in (32, 256):
        got = rc.rc_opportunity(a.t_ns, a.route, panel.n_labels, K, 50_000_000, 0)
        want = _want(a.t_ns, a.route, panel.n_labels, K, 50_000_000, 0)
        assert (got["fixed"], got["exact"], got["upper"]) == (want["fixed"], want["exact"], want["upper"]), K


@pytest.mark.parametrize("n,K,spacing,delta", [(40, 4, 3, 20), (40, 4, 7, 20), (9, 5, 1, 8), (100, 10, 2, 37)])
def test_evenly_spaced_closed_form(rc, n, K, spacing, delta):
    # n arrivals spaced evenly on one route: a delta-window holds m = floor(delta/spacing) + 1
    # events, and when m >= 2K - 1 every event can be batched (P* = n) if n >= K
    t = np.arange(n, dtype=np.int64) * spacing
    got = rc.rc_opportunity(t, np.zeros(n, np.uint32), 1, K, delta, 0)
    m = delta // spacing + 1
    if m >= 2 * K - 1 and n >= K:
        assert got["exact"] == n
    assert got == dict(n=n, **_want(t, np.zeros(n, np.uint32), 1, K, delta))


def test_threshold_one_serves_everything_and_empty_set(rc):
    t = np.array([5, 5, 9, 100], dtype=np.int64)
    assert rc.rc_opportunity(t, np.zeros(4, np.uint32), 1, 1, 3, 0) == dict(n=4, fixed=4, exact=4, upper=4)
    assert rc.rc_opportunity(np.zeros(0, np.int64), np.zeros(0, np.uint32), 1, 2, 3, 0) == dict(
        n=0, fixed=0, exact=0, upper=0)


def test_bad_arguments_are_rejected(rc):
    t = np.array([1, 2], dtype=np.int64)
    r = np.array([0, 1], dtype=np.uint32)
    for args in ((t, r, 2, 0, 5), (t, r, 2, 2, 0), (t, r, 1, 2, 5)):
        with pytest.raises(rc.RcError) as e:
            rc.rc_opportunity(*args)
        assert e.value.code == rc.RC_E_INVAL


def test_shares_and_ratios(rc):
    panel = wl.make_panel()
    a = wl.make_arrivals(10_000, panel)
    mem, _, _ = rc.form_cohorts(a.t_ns, a.route, a.session, panel.n_labels, 32, 50_000_000)
    got = rc.opportunity_shares(a.t_ns, a.route, panel.n_labels, 32, 50_000_000, mem.size)
    want = oracle.shares(a.t_ns, a.route, a.session, panel.n_labels, 32, 50_000_000)
    for k in ("F", "P", "U", "A", "G", "R_A"):
        assert got[k] == want[k], k
