"""Pins of the oracle's cohort-supply quantities: F (Eq. 2), U (Eqs. 3-4),
the exact assigned count behind P* (Eq. 6 / Algorithm 1) and the online
former behind A.

Independent references:
* subset brute force of Eq. 1 schedules on tiny inputs (arbitrary and equal
  relative deadlines, route-specific thresholds, boundary ties), as the paper
  checks its evaluator (Section 4, "Exact clock");
* Q_r(tau) evaluated at EVERY integer tau of [t_i, d_i] for U;
* closed forms on evenly spaced arrivals;
* hand-worked fixtures (tests/golden/shares_worked.json, former_worked.json);
* Proposition 1 (F <= P* <= U, A <= P*) and the five validity gates of
  Section 5.3 on replayed synthetic arrivals.
"""
import json
import os

import numpy as np
import pytest

import oracle
import rc_workload as wl
from conftest import GOLDEN


# ------------------------------------------------------------ brute force

def brute_exact(t, r, d, Kr):
    """Maximum number of events covered by disjoint Eq. 1 batches: a batch is
    a set of one route with size >= K_r that admits a launch time tau with
    t_i <= tau <= d_i for all members (i.e. max t <= min d).  Subset DP."""
    n = len(t)
    full = (1 << n) - 1
    feas = [False] * (1 << n)
    for mask in range(1, 1 << n):
        mem = [i for i in range(n) if mask >> i & 1]
        rr = {r[i] for i in mem}
        if len(rr) != 1:
            continue
        route = rr.pop()
        if len(mem) < Kr[route]:
            continue
        if max(t[i] for i in mem) <= min(d[i] for i in mem):
            feas[mask] = True
    best = [0] * (1 << n)
    for mask in range(1, 1 << n):
        low = (mask & -mask)
        rest = mask ^ low
        b = best[rest]
        sub = rest
        while True:
            B = sub | low
            if feas[B]:
                v = bin(B).count("1") + best[mask ^ B]
                if v > b:
                    b = v
            if sub == 0:
                break
            sub = (sub - 1) & rest
        best[mask] = b
    return best[full]


def brute_upper(t, r, delta, Kr):
    """Eq. 4 with Q evaluated at every integer tau in [t_i, t_i + delta]."""
    n = len(t)
    cnt = 0
    for i in range(n):
        best = 0
        for tau in range(t[i], t[i] + delta + 1):
            q = sum(1 for j in range(n) if r[j] == r[i] and t[j] <= tau <= t[j] + delta)
            best = max(best, q)
        cnt += best >= Kr[r[i]]
    return cnt


def _tiny_instances(seed, count):
    rng = np.random.default_rng(seed)
    for _ in range(count):
        n = int(rng.integers(1, 10))
        R = int(rng.integers(1, 4))
        delta = int(rng.integers(0, 7))
        span = int(rng.integers(1, 16))
        t = rng.integers(0, span, size=n).astype(np.int64)
        r = rng.integers(0, R, size=n).astype(np.uint32)
        Kr = rng.integers(1, 4, size=R).astype(np.uint32)
        yield t, r, R, Kr, delta


@pytest.mark.parametrize("seed", [1, 2, 3, 4])
def test_exact_count_matches_subset_brute_force(seed):
    for t, r, R, Kr, delta in _tiny_instances(seed, 60):
        d = t + delta
        want = brute_exact(list(t), list(r), list(d), list(Kr))
        got, bo, nb = oracle.exact_count(t, r, R, Kr, delta, method=0, want_witness=True)
        assert got == want, (t, r, Kr, delta)
        assert oracle.exact_count(t, r, R, Kr, delta, method=1) == want
        _check_witness(t, r, Kr, delta, bo, nb, got)


def _check_witness(t, r, Kr, delta, bo, nb, total):
    assert int((bo >= 0).sum()) == total
    assert set(int(b) for b in bo[bo >= 0]) == set(range(nb))
    for b in range(nb):
        mem = np.nonzero(bo == b)[0]
        assert len(set(int(x) for x in r[mem])) == 1
        route = int(r[mem[0]])
        assert len(mem) >= Kr[route]
        assert t[mem].max() - t[mem].min() <= delta
        # Lemma 1: a block is contiguous among its route's events sorted by (t, id)
        same = np.nonzero(r == route)[0]
        order = same[np.lexsort((same, t[same]))]
        pos = np.nonzero(np.isin(order, mem))[0]
        assert pos.max() - pos.min() + 1 == len(mem)


def test_brute_force_rejects_arbitrary_deadline_shortcuts():
    # with unequal deadlines the same releases can lose a batch: the brute
    # force follows Eq. 1 directly (tau must sit inside every [t_i, d_i])
    assert brute_exact([0, 1, 2], [0, 0, 0], [5, 1, 5], [3]) == 0
    assert brute_exact([0, 1, 2], [0, 0, 0], [5, 2, 5], [3]) == 3


@pytest.mark.parametrize("seed", [5, 6])
def test_upper_count_matches_every_tau_brute_force(seed):
    for t, r, R, Kr, delta in _tiny_instances(seed, 50):
        want = brute_upper(list(t), list(r), delta, list(Kr))
        got, el = oracle.upper_count(t, r, R, Kr, delta, want_eligible=True)
        assert got == want and int(el.sum()) == got


def test_worked_share_fixtures():
    cases = json.load(open(os.path.join(GOLDEN, "shares_worked.json")))["cases"]
    for c in cases:
        t = np.array(c["t"], np.int64)
        r = np.array(c["route"], np.uint32)
        Kr = c.get("Kr", c.get("K"))
        assert oracle.fixed_count(t, r, c["R"], Kr, c["delta"]) == c["F"], c["name"]
        assert oracle.exact_count(t, r, c["R"], Kr, c["delta"]) == c["P"], c["name"]
        assert oracle.exact_count(t, r, c["R"], Kr, c["delta"], method=1) == c["P"], c["name"]
        assert oracle.upper_count(t, r, c["R"], Kr, c["delta"]) == c["U"], c["name"]


# ------------------------------------------------------------ closed forms

@pytest.mark.parametrize("n,K,spacing,delta", [
    (50, 4, 3, 10), (50, 4, 3, 9), (51, 5, 2, 7), (10, 6, 1, 4), (100, 8, 5, 60), (7, 7, 1, 6),
    (40, 3, 10, 19), (40, 3, 10, 20),
])
def test_evenly_spaced_closed_forms(n, K, spacing, delta):
    t = np.arange(n, dtype=np.int64) * spacing
    r = np.zeros(n, np.uint32)
    m = delta // spacing + 1               # events that fit in one span of delta
    want_p = min(n, (n // K) * m) if m >= K else 0
    want_u = n if (m >= K and n >= K) else 0
    assert oracle.exact_count(t, r, 1, K, delta) == want_p
    assert oracle.upper_count(t, r, 1, K, delta) == want_u
    # fixed windows of width w = spacing * q hold q events each (origin 0)
    q = 4
    w = spacing * q
    full, rem = divmod(n, q)
    want_f = full * q * (q >= K) + rem * (rem >= K)
    assert oracle.fixed_count(t, r, 1, K, w) == want_f


def test_threshold_one_and_simultaneous_arrivals():
    rng = np.random.default_rng(3)
    t = rng.integers(0, 10**9, size=500).astype(np.int64)
    r = rng.integers(0, 5, size=500).astype(np.uint32)
    for f in (oracle.fixed_count, oracle.exact_count, oracle.upper_count):
        assert f(t, r, 5, 1, 1000) == 500
    t = np.full(40, 123, np.int64)
    r = np.zeros(40, np.uint32)
    for f in (oracle.fixed_count, oracle.exact_count, oracle.upper_count):
        assert f(t, r, 1, 40, 1) == 40
        assert f(t, r, 1, 41, 10) == 0
    assert oracle.exact_count(t, r, 1, 40, 0) == 40 and oracle.upper_count(t, r, 1, 40, 0) == 40


def test_zero_events():
    e = np.zeros(0, np.int64)
    z = np.zeros(0, np.uint32)
    assert oracle.fixed_count(e, z, 3, 2, 10) == 0
    assert oracle.exact_count(e, z, 3, 2, 10) == 0
    assert oracle.upper_count(e, z, 3, 2, 10) == 0
    mem, tau, cr = oracle.former(e, z, z, 3, 2, 10)
    assert mem.shape == (0, 2)


# ------------------------------------------------------------------ former

def test_former_worked_fixture():
    fx = json.load(open(os.path.join(GOLDEN, "former_worked.json")))
    ev = fx["events"]
    t = np.array([e["t"] for e in ev], np.int64)
    r = np.array([e["route"] for e in ev], np.uint32)
    s = np.array([e["session"] for e in ev], np.uint32)
    mem, tau, cr = oracle.former(t, r, s, fx["R"], fx["K"], fx["delta"])
    assert mem.tolist() == fx["cohorts"]
    assert tau.tolist() == fx["tau"]
    assert mem.size == fx["A_count"]


def test_gap_closure_and_online_ratio_worked_by_hand():
    """G (Eq. 7) and R_A (Eq. 9) on counts worked out by hand (K = 2,
    delta = 10, windows from origin 0).  Route 0 is the former fixture's
    events: windows [0,10) and [30,40) hold 3 and 2 -> F = 5; blocks {0,5,8}
    and one of {20,30} / {30,31} (a block of three would span 11) -> P = 5;
    every event shares some interval with another -> U = 6; the former
    launches {0,8} and {20,30} -> A = 4.  Route 1 is one pair {9,10} split by
    the window boundary: F = 0, P = U = A = 2.  Together F, P, U, A = 5, 7,
    8, 6: G = (7 - 5) / (8 - 5) = 2/3, R_A = (6 - 5) / (7 - 5) = 1/2.  Route 0
    alone has P = F: G = 0, R_A undefined."""
    t = np.array([0, 5, 8, 9, 10, 20, 30, 31], np.int64)
    r = np.array([0, 0, 0, 1, 1, 0, 0, 0], np.uint32)
    s = np.array([1, 1, 2, 6, 7, 3, 4, 5], np.uint32)
    sh = oracle.shares(t, r, s, 2, 2, 10)
    assert sh["counts"] == dict(F=5, P=7, U=8, A=6)
    assert sh["G"] == pytest.approx(2 / 3, abs=1e-15)
    assert sh["R_A"] == pytest.approx(0.5, abs=1e-15)
    only0 = r == 0
    sh0 = oracle.shares(t[only0], r[only0], s[only0], 1, 2, 10)
    assert sh0["counts"] == dict(F=5, P=5, U=6, A=4)
    assert sh0["G"] == 0.0 and sh0["R_A"] is None


def _check_former(t, r, s, K, delta, mem, tau, cr):
    used = mem.reshape(-1)
    assert len(np.unique(used)) == len(used)                 # each event at most once
    for c in range(len(mem)):
        m = mem[c]
        assert len(np.unique(s[m])) == K                    # distinct sessions
        assert np.all(r[m] == cr[c])                        # one route (Eq. 1)
        assert np.all(t[m] <= tau[c]) and np.all(tau[c] <= t[m] + delta)  # Eq. 1 window
        assert tau[c] in set(int(x) for x in t[m])          # launched on an arrival
    assert np.all(np.diff(tau) >= 0)                        # launch order


@pytest.mark.parametrize("C,K", [(2000, 4), (5000, 16), (5000, 64)])
def test_former_feasible_and_below_exact(C, K):
    panel = wl.make_panel()
    a = wl.make_arrivals(C, panel, horizon_s=6.0)
    delta = 50_000_000
    mem, tau, cr = oracle.former(a.t_ns, a.route, a.session, panel.n_labels, K, delta)
    _check_former(a.t_ns, a.route, a.session, K, delta, mem, tau, cr)
    assert mem.size <= oracle.exact_count(a.t_ns, a.route, panel.n_labels, K, delta)


def test_former_small_random_against_brute_force():
    rng = np.random.default_rng(11)
    for _ in range(80):
        n = int(rng.integers(1, 10))
        t = np.sort(rng.integers(0, 12, size=n)).astype(np.int64)
        r = rng.integers(0, 2, size=n).astype(np.uint32)
        s = rng.integers(0, 4, size=n).astype(np.uint32)
        K = int(rng.integers(1, 4))
        delta = int(rng.integers(0, 6))
        mem, tau, cr = oracle.former(t, r, s, 2, K, delta)
        _check_former(t, r, s, K, delta, mem, tau, cr)
        assert mem.size <= brute_exact(list(t), list(r), list(t + delta), [K, K])


# --------------------------------------------------- Prop. 1 and the gates

def _replay(C, horizon_s=6.0, seed_index=0):
    panel = wl.make_panel()
    return panel, wl.make_arrivals(C, panel, horizon_s=horizon_s, seed_index=seed_index)


def _all_three(t, r, R, K, delta):
    return (oracle.fixed_count(t, r, R, K, delta), oracle.exact_count(t, r, R, K, delta),
            oracle.upper_count(t, r, R, K, delta))


@pytest.mark.parametrize("C", [3000, 20000])
def test_five_validity_gates_on_replay(C):
    panel, a = _replay(C)
    R = panel.n_labels
    groupings = [
        ("route", a.route, R),
        ("class", (a.route % 8).astype(np.uint32), 8),
        ("pooled", np.zeros_like(a.route), 1),
    ]
    deltas = [10_000_000, 25_000_000, 50_000_000, 100_000_000, 250_000_000]
    Ks = [32, 64, 128, 256]
    res = {}
    for gname, r, RR in groupings:
        for dl in deltas:
            for K in Ks:
                f, p, u = _all_three(a.t_ns, r, RR, K, dl)
                res[gname, dl, K] = (f, p, u)
                assert f <= p <= u                                     # Prop. 1
                if f == u:
                    assert p == f                                      # gate 5
    for dl in deltas:
        for K in Ks:
            for fine, coarse in (("route", "class"), ("class", "pooled")):
                for q in range(3):                                     # gate 2: coarsening
                    assert res[fine, dl, K][q] <= res[coarse, dl, K][q]
    for g, _, _ in groupings:
        for K in Ks:
            for d0, d1 in zip(deltas, deltas[1:]):                     # gate 3: wider deadline
                assert res[g, d0, K][1] <= res[g, d1, K][1]
                assert res[g, d0, K][2] <= res[g, d1, K][2]
                if d1 % d0 == 0:                                       # nested windows
                    assert res[g, d0, K][0] <= res[g, d1, K][0]
        for dl in deltas:
            for K0, K1 in zip(Ks, Ks[1:]):                             # gate 4: larger threshold
                for q in range(3):
                    assert res[g, dl, K1][q] <= res[g, dl, K0][q]


def test_online_share_below_exact_share():
    panel, a = _replay(20000)
    sh = oracle.shares(a.t_ns, a.route, a.session, panel.n_labels, 32, 50_000_000)
    assert sh["A"] <= sh["P"] <= sh["U"] and sh["F"] <= sh["P"]
    assert sh["counts"]["A"] % 32 == 0


def test_shares_do_not_depend_on_input_order():
    panel, a = _replay(3000, horizon_s=3.0)
    perm = np.random.default_rng(5).permutation(a.n)
    for K in (8, 32):
        base = _all_three(a.t_ns, a.route, panel.n_labels, K, 50_000_000)
        shuf = _all_three(a.t_ns[perm], a.route[perm], panel.n_labels, K, 50_000_000)
        assert base == shuf


def test_fixed_windows_floor_toward_minus_infinity_and_follow_origin():
    # windows [o + w*delta, o + (w+1)*delta): with origin 0 and delta 10,
    # -5 and -1 share window -1 while 3 sits in window 0 (hand-worked)
    t = np.array([-5, -1, 3], np.int64)
    r = np.zeros(3, np.uint32)
    assert oracle.fixed_count(t, r, 1, 2, 10) == 2
    # shifting the origin to -6 puts all three in [-6, 4)
    assert oracle.fixed_count(t, r, 1, 3, 10, origin=-6) == 3
    assert oracle.fixed_count(t, r, 1, 3, 10, origin=0) == 0
