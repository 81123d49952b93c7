"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle, bit
for bit, on every decision, effect, per-step state record and final state
(the exactness contract of Sections 2.2 and 7.3), for every mechanism of
Section 7.1 / 8.1 and every workload shape."""
import importlib

import numpy as np
import pytest

import rc_workload as wl

pytestmark = pytest.mark.gpu

MECHS = ("host_rt", "resident_cond", "resident_persist", "fixed_nested", "floor")


@pytest.fixture(scope="module")
def g():
    return importlib.import_module("gpu_util")


@pytest.fixture(scope="module")
def rc():
    return importlib.import_module("paper_2608_12123_gb300")


def _inputs(cfg, K, S, SB, P, n_sets, N=None):
    tables = wl.make_tables(S, wl.stream_seed(cfg, wl.Purpose.TABLE))
    Nn = K if N is None else N
    state0 = wl.make_state(Nn, S, SB, wl.stream_seed(cfg, wl.Purpose.STATE))
    outc, pay, idx = wl.make_cohort_events(cfg, n_sets, K, P, n_sessions=N)
    return tables, state0, outc, pay, idx


def _check_all(g, rc, mechs, tables, state0, outc, pay, idx, n_steps, K, sel0=0, log=True, what=""):
    want = g.run_oracle(tables, state0, outc, pay, idx, n_steps, sel0=sel0, log=log)
    for name in mechs:
        mech = rc.MECHANISMS[name]
        got = g.run_gpu(mech, tables, state0, outc, pay, idx, n_steps, K, sel0=sel0, log=log,
                        floor_seq=want["decisions"])
        w = dict(want)
        if name == "floor":
            w.pop("sel")  # the floor replays the sequence and leaves the flag alone
        g.assert_same(got, w, f"{what} {name}")
    return want


def test_tiny_chain_all_mechanisms(g, rc):
    # K = 32, S = 16, 16-byte records, 32-byte payloads, 1,000 chained steps
    K, S, SB, P, n = 32, 16, 16, 32, 1000
    tables, state0, outc, pay, idx = _inputs(1, K, S, SB, P, n)
    want = _check_all(g, rc, MECHS, tables, state0, outc, pay, idx, n, K, what="tiny chain")
    assert 0 < want["decisions"].sum() < n  # both route bodies are exercised


@pytest.mark.parametrize("SB,P", [(16, 32), (16, 64), (16, 128), (64, 32), (64, 64), (64, 128)])
@pytest.mark.parametrize("K", [1, 7, 33, 255, 257, 1000, 1025, 3001])
def test_ragged_shapes(g, rc, SB, P, K):
    N = 4 * K + 5
    S = 256 if SB == 64 else 32
    n = 6
    tables, state0, outc, pay, idx = _inputs(40 + K % 7, K, S, SB, P, 4, N=N)
    _check_all(g, rc, ("host_rt", "resident_cond", "resident_persist", "fixed_nested"), tables, state0, outc,
               pay, idx, n, K, sel0=K & 1, what=f"K={K} SB={SB} P={P}")


def test_floor_multi_cta_and_identity(g, rc):
    K, S, SB, P, n = 700, 64, 64, 64, 12
    tables, state0, outc, pay, idx = _inputs(7, K, S, SB, P, n)
    _check_all(g, rc, MECHS, tables, state0, outc, pay, idx, n, K, what="identity K=700")


def test_empty_cohort_and_zero_steps(g, rc):
    tables, state0, outc, pay, idx = _inputs(3, 4, 16, 16, 32, 1, N=8)
    for name in ("host_rt", "resident_persist", "resident_cond"):
        got = g.run_gpu(rc.MECHANISMS[name], tables, state0, outc[:, :0], pay[:, :0], idx[:, :0], 5, 0, sel0=1)
        assert np.array_equal(got["decisions"], np.zeros(5, np.uint32))
        assert np.array_equal(got["state"], state0) and got["sel"] == 0
        got = g.run_gpu(rc.MECHANISMS[name], tables, state0, outc, pay, idx, 0, 4, sel0=1, log=False)
        assert np.array_equal(got["state"], state0) and got["sel"] == 1


def test_host_buffers_give_identical_results(g, rc):
    K, S, SB, P, n = 300, 64, 16, 64, 20
    tables, state0, outc, pay, idx = _inputs(9, K, S, SB, P, n, N=1000)
    want = g.run_oracle(tables, state0, outc, pay, idx, n)
    for name in ("host_rt", "resident_persist", "resident_cond"):
        got = g.run_gpu(rc.MECHANISMS[name], tables, state0, outc, pay, idx, n, K, host_buffers=True)
        g.assert_same(got, want, f"host buffers {name}")


@pytest.mark.parametrize("K,N,n,SB,P,identity", [(256, 300, 128, 16, 64, False), (256, 259, 1000, 16, 64, False),
                                                   (64, 70, 400, 64, 128, False), (40, 40, 330, 16, 32, True),
                                                   (2048, 2100, 130, 16, 64, False), (8192, 1 << 20, 129, 64, 128, False)])
def test_host_buffers_in_pieces(g, rc, K, N, n, SB, P, identity):
    """A persistent chain over host-memory events, one cohort per step, runs in
    pieces (64 steps, then four times the previous up to 1,024) with the
    copies of later pieces overlapping the current one; sessions recur across the piece
    boundaries (N close to K).  Every output equals the oracle's, and the
    whole chain counts two launches per piece where a link pass precedes the
    chain."""
    import torch
    S = 256 if SB == 64 else 64
    tables, state0, outc, pay, idx = _inputs(110 + K % 11 + n, K, S, SB, P, n, N=N)
    if identity:
        idx = None
    want = g.run_oracle(tables, state0, outc, pay, idx, n, sel0=1)
    got = g.run_gpu(rc.RC_MECH_RESIDENT_PERSIST, tables, state0, outc, pay, idx, n, K, sel0=1, host_buffers=True)
    g.assert_same(got, want, f"pieces K={K} N={N} n={n}")
    pieces, first, size = 0, 0, 64
    while first < n:
        first += min(size, n - first)
        size = min(4 * size, 1024)
        pieces += 1
    ctx = rc.rc_init(S, tables, SB, P, K, N, torch.cuda.current_stream())
    try:
        state = g.dev(state0.copy())
        ev = rc.make_events(np.ascontiguousarray(outc), np.ascontiguousarray(pay),
                            None if idx is None else np.ascontiguousarray(idx), payload_bytes=P, n_sets=n)
        dec = np.zeros(n, np.uint32)
        rc.rc_chain(ctx, n, rc.RC_MECH_RESIDENT_PERSIST, state, ev, K, dec)
        _, launches = rc.rc_last_chain_stats(ctx)
        # per piece: its step base, then the chain (with its pre-pass); one
        # more write returns the step base to 0
        per_piece = (launches - 1) // pieces
        assert launches == per_piece * pieces + 1 and per_piece in (2, 3, 4), (launches, pieces)
    finally:
        rc.rc_free(ctx)


def test_error_step_counts_from_the_chain_start_in_pieces(g, rc):
    """A latched error in a later piece reports its step in the whole chain."""
    K, S, SB, P, n = 64, 16, 16, 32, 200
    tables, state0, outc, pay, idx = _inputs(131, K, S, SB, P, n, N=500)
    o2 = outc.copy()
    o2[150, 7] = 8  # step 150 lies in the second piece (64 + 256 + ...)
    with pytest.raises(rc.RcError) as e:
        g.run_gpu(rc.RC_MECH_RESIDENT_PERSIST, tables, state0, o2, pay, idx, n, K, host_buffers=True)
    assert e.value.code == rc.RC_E_STATE
    assert "step 150, member 7" in str(e.value), str(e.value)


def test_cohort_step_api_carries_the_flag_and_checks_deadlines(g, rc):
    import torch
    K, S, SB, P, n = 100, 32, 16, 32, 25
    tables, state0, outc, pay, idx = _inputs(11, K, S, SB, P, n, N=400)
    want = g.run_oracle(tables, state0, outc, pay, idx, n)
    ctx = rc.rc_init(S, tables, SB, P, K, 400, torch.cuda.current_stream())
    try:
        state = g.dev(state0.copy())
        for j in range(n):
            ev = rc.make_events(g.dev(outc[j]), g.dev(pay[j]), g.dev(idx[j]), n_sets=1, launch_ns=1000 + j)
            eff = torch.zeros(K * 16, dtype=torch.uint8, device="cuda")
            if j == 3:
                with pytest.raises(rc.RcError) as e:
                    rc.rc_cohort_step(ctx, state, ev, K, 1000 + j - 1, eff)
                assert e.value.code == rc.RC_E_DEADLINE
            rc.rc_cohort_step(ctx, state, ev, K, 1000 + j, eff)
            assert np.array_equal(g.host(eff, np.uint8).reshape(K, 16), want["effects"][j])
            assert rc.rc_get_decision(ctx) == want["decisions"][j]
        rc.rc_sync(ctx)
        assert np.array_equal(g.host(state, np.uint8).reshape(state0.shape), want["state"])
    finally:
        rc.rc_free(ctx)


def test_bad_inputs_are_latched_and_the_context_survives(g, rc):
    import torch
    K, S, SB, P, n = 64, 16, 16, 32, 3
    tables, state0, outc, pay, idx = _inputs(13, K, S, SB, P, n, N=200)
    cases = []
    o2 = outc.copy(); o2[1, 5] = 8
    cases.append(("outcome", state0, o2, idx, rc.RC_E_STATE))
    s2 = state0.copy(); s2[idx[0, 9], 0:4] = np.frombuffer(np.uint32(S).tobytes(), np.uint8)
    cases.append(("state", s2, outc, idx, rc.RC_E_STATE))
    i2 = idx.copy(); i2[2, 17] = 200
    cases.append(("index", state0, outc, i2, rc.RC_E_INDEX))
    for name in ("host_rt", "resident_persist", "resident_cond", "fixed_nested"):
        for what, st, oc, ix, code in cases:
            with pytest.raises(rc.RcError) as e:
                g.run_gpu(rc.MECHANISMS[name], tables, st, oc, pay, ix, n, K)
            assert e.value.code == code, (name, what)
    # the device stays usable: a clean chain right after matches the oracle
    want = g.run_oracle(tables, state0, outc, pay, idx, n)
    g.assert_same(g.run_gpu(rc.RC_MECH_RESIDENT_PERSIST, tables, state0, outc, pay, idx, n, K), want, "after errors")


@pytest.mark.parametrize("what", ["outcome", "state", "index"])
@pytest.mark.parametrize("K,identity", [(64, False), (256, False), (32, True)])
def test_bad_inputs_in_two_step_chains(g, rc, what, K, identity):
    """The chains that key two steps per block barrier (explicit sessions, 64
    steps or more; identity sessions) latch a bad input with the step it sits
    in and keep the context usable; a clean chain right after matches the
    oracle."""
    S, SB, P, n = 16, 16, 32, 70
    tables, state0, outc, pay, idx = _inputs(150 + K, K, S, SB, P, n, N=None if identity else 4 * K)
    if identity:
        idx = None
    st, oc, ix = state0.copy(), outc.copy(), None if idx is None else idx.copy()
    bad_step, bad_member = 45, 5
    if what == "outcome":
        oc[bad_step, bad_member] = 8
        code = rc.RC_E_STATE
    elif what == "state":
        sess = bad_member if identity else int(idx[0, bad_member])
        st[sess, 0:4] = np.frombuffer(np.uint32(S).tobytes(), np.uint8)
        bad_step, code = 0, rc.RC_E_STATE
    else:
        if identity:
            pytest.skip("identity sessions have no index array")
        ix[bad_step, bad_member] = 4 * K
        code = rc.RC_E_INDEX
    with pytest.raises(rc.RcError) as e:
        g.run_gpu(rc.RC_MECH_RESIDENT_PERSIST, tables, st, oc, pay, ix, n, K)
    assert e.value.code == code
    assert f"step {bad_step}," in str(e.value), str(e.value)
    want = g.run_oracle(tables, state0, outc, pay, idx, n)
    g.assert_same(g.run_gpu(rc.RC_MECH_RESIDENT_PERSIST, tables, state0, outc, pay, idx, n, K), want,
                  f"after {what}")


def test_grid_barrier_wait_is_bounded(g, rc, monkeypatch):
    """A CTA that never arrives (test hook) makes the others' bounded waits run
    out: RC_E_TIMEOUT comes back and the context keeps working."""
    import torch
    monkeypatch.setenv("RC_NO_CLUSTER", "1")  # the grid kernel, not the cluster one
    K, S, SB, P, n = 4096, 16, 16, 32, 4
    tables, state0, outc, pay, idx = _inputs(17, K, S, SB, P, 2, N=5000)
    ctx = rc.rc_init(S, tables, SB, P, K, 5000, torch.cuda.current_stream())
    try:
        rc.rc_set_wait_limits(ctx, 2_000_000, 30_000_000_000)  # 2 ms device waits
        state = g.dev(state0.copy())
        ev = rc.make_events(g.dev(outc), g.dev(pay), g.dev(idx))
        dec = torch.zeros(n, dtype=torch.int32, device="cuda")
        rc.rc_debug_skip_arrival(ctx, True)
        with pytest.raises(rc.RcError) as e:
            rc.rc_chain(ctx, n, rc.RC_MECH_RESIDENT_PERSIST, state, ev, K, dec)
        assert e.value.code == rc.RC_E_TIMEOUT
        # hook disarmed: the same context runs a clean chain
        state = g.dev(state0.copy())
        rc.rc_set_decision(ctx, 0)
        rc.rc_chain(ctx, n, rc.RC_MECH_RESIDENT_PERSIST, state, ev, K, dec)
        want = g.run_oracle(tables, state0, outc, pay, idx, n, log=False)
        assert np.array_equal(g.host(dec, np.uint32), want["decisions"])
        assert np.array_equal(g.host(state, np.uint8).reshape(state0.shape), want["state"])
    finally:
        rc.rc_free(ctx)


def test_launch_floor_probes_run(g, rc):
    """Every launch-floor probe returns a positive time (kind 4: empty grid
    steps over one CTA per SM, each wait bounded at 2 ms); an unknown kind is
    refused; the context then still runs a chain bit-exactly."""
    import torch
    K, S, SB, P, n = 32, 16, 16, 32, 6
    tables, state0, outc, pay, _ = _inputs(1, K, S, SB, P, n)
    ctx = rc.rc_init(S, tables, SB, P, K, K, torch.cuda.current_stream())
    try:
        rc.rc_set_wait_limits(ctx, 2_000_000, 30_000_000_000)
        for kind in (0, 1, 2, 3, 4):
            us = rc.rc_launch_floor(ctx, kind, 200)
            assert 0.0 < us < 1000.0
        with pytest.raises(rc.RcError) as e:
            rc.rc_launch_floor(ctx, 5, 10)
        assert e.value.code == rc.RC_E_INVAL
        want = g.run_oracle(tables, state0, outc, pay, None, n)
        state = g.dev(state0.copy())
        ev = rc.make_events(g.dev(outc), g.dev(pay), None, payload_bytes=P, n_sets=n)
        dec = torch.zeros(n, dtype=torch.int32, device="cuda")
        rc.rc_chain(ctx, n, rc.RC_MECH_RESIDENT_PERSIST, state, ev, K, dec)
        assert np.array_equal(g.host(dec, np.uint32), want["decisions"])
        assert np.array_equal(g.host(state, np.uint8).reshape(state0.shape), want["state"])
    finally:
        rc.rc_free(ctx)


@pytest.mark.parametrize("kernel", ["gpair", "link"])
@pytest.mark.parametrize("n_sets", [1, 2, 3, 4, 7])
@pytest.mark.parametrize("SB,P,K,N", [(64, 128, 2056, 2100), (16, 64, 4104, 12000), (64, 32, 1032, 1032)])
def test_grid_link_records_stored_early_and_late(g, rc, monkeypatch, kernel, n_sets, SB, P, K, N):
    """The grid chains over many steps: sessions recurring at distances 1, 2,
    3 and more (rings of 1 to 7 cohorts drawn from N near K) must see every
    earlier record.  "link" (one step per barrier): through the linked gather
    after the barrier or the unlinked gather run ahead while it is awaited;
    "gpair" (two steps per barrier): through the input-state ring, the
    second link of an odd step whose session is in the even one, the record
    handed from the even step to the odd one, or the state array."""
    monkeypatch.setenv("RC_NO_CLUSTER", "1")
    monkeypatch.setenv("RC_GRID_PAIR", "1" if kernel == "gpair" else "0")
    S = 256 if SB == 64 else 64
    tables, state0, outc, pay, idx = _inputs(140 + n_sets + K % 7, K, S, SB, P, n_sets, N=N)
    n = 14
    want = g.run_oracle(tables, state0, outc, pay, idx, n, sel0=1)
    got = g.run_gpu(rc.RC_MECH_RESIDENT_PERSIST, tables, state0, outc, pay, idx, n, K, sel0=1)
    g.assert_same(got, want, f"grid {kernel} n_sets={n_sets} SB={SB} P={P} K={K} N={N}")


@pytest.mark.parametrize("n", [1, 2, 3, 4, 5, 13])
@pytest.mark.parametrize("n_sets", [1, 2, 5])
@pytest.mark.parametrize("SB,P", [(16, 32), (64, 128)])
def test_grid_pair_step_counts(g, rc, monkeypatch, n, n_sets, SB, P):
    """Two steps per grid barrier on chains of odd and even length, the
    shortest among them (a region with one key step, a last region that only
    completes), sessions recurring at every distance (N near K)."""
    monkeypatch.setenv("RC_NO_CLUSTER", "1")
    monkeypatch.setenv("RC_GRID_PAIR", "1")
    K, N = 2056, 2300
    S = 256 if SB == 64 else 64
    tables, state0, outc, pay, idx = _inputs(170 + n + 7 * n_sets, K, S, SB, P, n_sets, N=N)
    want = g.run_oracle(tables, state0, outc, pay, idx, n, sel0=n & 1)
    got = g.run_gpu(rc.RC_MECH_RESIDENT_PERSIST, tables, state0, outc, pay, idx, n, K, sel0=n & 1)
    g.assert_same(got, want, f"grid pair n={n} n_sets={n_sets} SB={SB} P={P}")


@pytest.mark.parametrize("what", ["state_even", "state_odd", "outcome_even", "outcome_odd", "index_odd"])
def test_grid_pair_errors_report_the_earlier_step(g, rc, monkeypatch, what):
    """Two steps keyed in one region by different CTAs: a bad state first met
    in the even step and carried into the odd one is reported at the even
    step; a bad outcome or index is reported at its own step."""
    monkeypatch.setenv("RC_NO_CLUSTER", "1")
    monkeypatch.setenv("RC_GRID_PAIR", "1")
    K, S, SB, P, n, N = 4104, 64, 16, 64, 6, 4400
    tables, state0, outc, pay, idx = _inputs(190, K, S, SB, P, n, N=N)
    st, oc, ix = state0.copy(), outc.copy(), idx.copy()
    even = what.endswith("even")
    if what.startswith("state"):
        # the session's first step in the chain: step 0, its session also in
        # step 1 (carried into the odd step); or step 1, its session not in 0
        j = 0 if even else 1
        pick = np.isin(idx[0], idx[1]) if even else ~np.isin(idx[1], idx[0])
        m = int(np.flatnonzero(pick)[0])
        st[int(idx[j, m]), 0:4] = np.frombuffer(np.uint32(S + 3).tobytes(), np.uint8)
        code = rc.RC_E_STATE
    else:
        # step 2 with its session also in step 3, or step 3 with it in step 2
        j = 2 if even else 3
        m = int(np.flatnonzero(np.isin(idx[j], idx[j + 1] if even else idx[j - 1]))[0])
        if what.startswith("outcome"):
            oc[j, m] = 9
            code = rc.RC_E_STATE
        else:
            ix[j, m] = N + 5
            code = rc.RC_E_INDEX
    with pytest.raises(rc.RcError) as e:
        g.run_gpu(rc.RC_MECH_RESIDENT_PERSIST, tables, st, oc, pay, ix, n, K)
    assert e.value.code == code
    assert f"step {j}," in str(e.value), str(e.value)


@pytest.mark.parametrize("what", ["state_first", "outcome_linked", "outcome_forward", "index"])
def test_grid_link_errors_report_their_step(g, rc, monkeypatch, what):
    """The grid chain split by links keys a linked member from the state its
    session's previous step publishes: a bad state carried that way is
    reported at the step it was first met, a bad outcome of a linked member
    or of one whose session goes on into the next step at its own step, a bad
    index at its own step; a clean chain right after matches the oracle."""
    monkeypatch.setenv("RC_NO_CLUSTER", "1")
    monkeypatch.setenv("RC_GRID_PAIR", "0")
    monkeypatch.setenv("RC_NO_GRID_LINK", "0")
    K, S, SB, P, n, N = 4104, 64, 16, 64, 6, 4400
    tables, state0, outc, pay, idx = _inputs(210, K, S, SB, P, n, N=N)
    st, oc, ix = state0.copy(), outc.copy(), idx.copy()
    if what == "state_first":
        # a session of step 0 that is also in step 1 (its state reaches step 1 published)
        j = 0
        m = int(np.flatnonzero(np.isin(idx[0], idx[1]))[0])
        st[int(idx[0, m]), 0:4] = np.frombuffer(np.uint32(S + 3).tobytes(), np.uint8)
        code = rc.RC_E_STATE
    elif what == "outcome_linked":
        j = 2
        m = int(np.flatnonzero(np.isin(idx[2], idx[1]))[0])
        oc[j, m] = 9
        code = rc.RC_E_STATE
    elif what == "outcome_forward":
        j = 2
        m = int(np.flatnonzero(np.isin(idx[2], idx[3]) & ~np.isin(idx[2], idx[1]))[0])
        oc[j, m] = 9
        code = rc.RC_E_STATE
    else:
        j = 3
        m = int(np.flatnonzero(np.isin(idx[3], idx[2]))[0])
        ix[j, m] = N + 5
        code = rc.RC_E_INDEX
    with pytest.raises(rc.RcError) as e:
        g.run_gpu(rc.RC_MECH_RESIDENT_PERSIST, tables, st, oc, pay, ix, n, K)
    assert e.value.code == code
    assert f"step {j}," in str(e.value), str(e.value)
    want = g.run_oracle(tables, state0, outc, pay, idx, n, sel0=1)
    got = g.run_gpu(rc.RC_MECH_RESIDENT_PERSIST, tables, state0, outc, pay, idx, n, K, sel0=1)
    g.assert_same(got, want, f"grid link after {what}")


@pytest.mark.parametrize("kernel", ["gpair", "link", "owned", "split", "tma", "plain"])
@pytest.mark.parametrize("SB,P", [(16, 32), (16, 64), (64, 128), (64, 32)])
@pytest.mark.parametrize("K,N,identity", [(1032, 5000, False), (4104, 9001, False), (4104, 4200, False),
                                          (2048, 2048, True), (65536, 70000, False), (65536, 1 << 20, False)])
def test_persistent_grid_kernels(g, rc, monkeypatch, kernel, SB, P, K, N, identity):
    """The cooperative persistent kernels: split-phase (explicit sessions, K a
    multiple of 8), TMA-fed and plain, on member counts that do not split
    evenly over SMs, with sessions recurring from step to step (N near K);
    "link" is the grid chain split by links (the default for explicit
    sessions), "gpair" the grid chain keying two steps per barrier (opt-in),
    the others turn both off."""
    monkeypatch.setenv("RC_OWNED", "1" if kernel == "owned" else "0")
    monkeypatch.setenv("RC_SPLIT", "1" if kernel == "split" else "0")
    monkeypatch.setenv("RC_NO_TMA", "1" if kernel == "plain" else "0")
    monkeypatch.setenv("RC_NO_GRID_LINK", "0" if kernel == "link" else "1")
    monkeypatch.setenv("RC_GRID_PAIR", "1" if kernel == "gpair" else "0")
    monkeypatch.setenv("RC_NO_CLUSTER", "1")  # K <= 8192 would otherwise take the cluster kernel
    S = 256 if SB == 64 else 64
    tables, state0, outc, pay, idx = _inputs(50 + K % 11, K, S, SB, P, 3, N=None if identity else N)
    n = 5
    want = g.run_oracle(tables, state0, outc, pay, idx, n, sel0=1)
    got = g.run_gpu(rc.RC_MECH_RESIDENT_PERSIST, tables, state0, outc, pay, idx, n, K, sel0=1)
    g.assert_same(got, want, f"grid {kernel} K={K} N={N} SB={SB} P={P}")


@pytest.mark.parametrize("kernel", ["gpair", "link", "owned", "split", "tma", "plain"])
def test_grid_barrier_wait_is_bounded_every_grid_kernel(g, rc, monkeypatch, kernel):
    import torch
    monkeypatch.setenv("RC_OWNED", "1" if kernel == "owned" else "0")
    monkeypatch.setenv("RC_SPLIT", "1" if kernel == "split" else "0")
    monkeypatch.setenv("RC_NO_TMA", "1" if kernel == "plain" else "0")
    monkeypatch.setenv("RC_NO_GRID_LINK", "0" if kernel == "link" else "1")
    monkeypatch.setenv("RC_GRID_PAIR", "1" if kernel == "gpair" else "0")
    monkeypatch.setenv("RC_NO_CLUSTER", "1")  # K <= 8192 would otherwise take the cluster kernel
    K, S, SB, P, n = 8192, 16, 16, 64, 4
    tables, state0, outc, pay, idx = _inputs(19, K, S, SB, P, 2, N=9000)
    ctx = rc.rc_init(S, tables, SB, P, K, 9000, torch.cuda.current_stream())
    try:
        rc.rc_set_wait_limits(ctx, 2_000_000, 30_000_000_000)
        state = g.dev(state0.copy())
        ev = rc.make_events(g.dev(outc), g.dev(pay), g.dev(idx))
        dec = torch.zeros(n, dtype=torch.int32, device="cuda")
        rc.rc_debug_skip_arrival(ctx, True)
        with pytest.raises(rc.RcError) as e:
            rc.rc_chain(ctx, n, rc.RC_MECH_RESIDENT_PERSIST, state, ev, K, dec)
        assert e.value.code == rc.RC_E_TIMEOUT
        state = g.dev(state0.copy())
        rc.rc_set_decision(ctx, 0)
        rc.rc_chain(ctx, n, rc.RC_MECH_RESIDENT_PERSIST, state, ev, K, dec)
        want = g.run_oracle(tables, state0, outc, pay, idx, n, log=False)
        assert np.array_equal(g.host(dec, np.uint32), want["decisions"])
        assert np.array_equal(g.host(state, np.uint8).reshape(state0.shape), want["state"])
    finally:
        rc.rc_free(ctx)


@pytest.mark.parametrize("kernel", ["owned", "split", "pair", "prod", "link", "plain"])
@pytest.mark.parametrize("P", [32, 64, 128])
@pytest.mark.parametrize("K,N", [(8, 9), (64, 67), (64, 128), (256, 259), (256, 512), (256, 1500), (496, 1000),
                                 (512, 513), (100, 300), (256, 1 << 20)])
def test_small_cohort_repeated_sessions(g, rc, monkeypatch, kernel, P, K, N):
    """Sessions that recur in consecutive steps at other member positions: each
    persistent kernel must see the records the previous step wrote ("pair":
    the single-CTA chain keying two steps per barrier, taken where it applies,
    K <= 256 and P <= 64; "prod" with it turned off)."""
    monkeypatch.setenv("RC_OWNED", "1" if kernel == "owned" else "0")
    monkeypatch.setenv("RC_SPLIT", "1" if kernel == "split" else "0")
    monkeypatch.setenv("RC_NO_PIPE", "1" if kernel == "plain" else "0")
    monkeypatch.setenv("RC_NO_PROD", "1" if kernel == "link" else "0")
    monkeypatch.setenv("RC_NO_PAIR", "0" if kernel == "pair" else "1")
    tables, state0, outc, pay, idx = _inputs(60 + K % 13 + P, K, 64, 16, P, 40, N=N)
    n = 70 if kernel == "pair" else 40  # the pair chain serves chains of 64 steps or more
    want = g.run_oracle(tables, state0, outc, pay, idx, n, sel0=1)
    got = g.run_gpu(rc.RC_MECH_RESIDENT_PERSIST, tables, state0, outc, pay, idx, n, K, sel0=1)
    g.assert_same(got, want, f"{kernel} K={K} N={N} P={P}")


@pytest.mark.parametrize("n", [30, 31])
@pytest.mark.parametrize("mode", ["two", "one", "plain"])
@pytest.mark.parametrize("SB,P,K", [(16, 32, 32), (16, 32, 256), (64, 128, 256), (64, 64, 700), (16, 128, 1024),
                                    (16, 64, 500), (64, 32, 8)])
def test_single_cta_identity_sessions(g, rc, monkeypatch, mode, SB, P, K, n):
    """Member m = session m: the record stays in registers.  "two": two steps
    per block barrier (K <= 512), "one": one step per barrier, "plain": the
    plain single-CTA kernel.  An odd step count leaves a last region of one
    step."""
    monkeypatch.setenv("RC_NO_PIPE", "1" if mode == "plain" else "0")
    monkeypatch.setenv("RC_NO_PAIR", "1" if mode == "one" else "0")
    S = 256 if SB == 64 else 128
    tables, state0, outc, pay, idx = _inputs(80 + K % 17, K, S, SB, P, n)
    want = g.run_oracle(tables, state0, outc, pay, idx, n, sel0=n % 2)
    got = g.run_gpu(rc.RC_MECH_RESIDENT_PERSIST, tables, state0, outc, pay, idx, n, K, sel0=n % 2)
    g.assert_same(got, want, f"identity {mode} SB={SB} P={P} K={K} n={n}")


@pytest.mark.parametrize("kernel", ["pair", "prod"])
@pytest.mark.parametrize("n_sets", [1, 2, 3, 7])
@pytest.mark.parametrize("SB,P,K,extra,want_launches", [(16, 64, 256, 0, 2), (16, 64, 256, 1, 2), (16, 32, 7, 2, 2),
                                                   (64, 64, 256, 1, 2), (16, 128, 300, 3, 2), (64, 32, 33, 0, 2),
                                                   (16, 64, 264, 9, 2), (16, 64, 512, 5, 2), (64, 128, 512, 1, 1),
                                                   (64, 128, 64, 3, 2), (16, 32, 8, 0, 2), (16, 128, 248, 40, 2),
                                                   (64, 64, 64, 5, 2), (64, 32, 128, 9, 2), (64, 64, 128, 0, 2)])
def test_linked_single_cta_ring_wraps(g, rc, monkeypatch, SB, P, K, extra, want_launches, n_sets, kernel):
    """The single-CTA chains that take recurring sessions from shared rings:
    cohorts drawn from N = K + extra sessions, so nearly every session recurs
    in the next steps at another position, and a ring of 1, 2, 3 or 7 cohorts,
    so links wrap (with one cohort every member follows itself).  K a
    multiple of 8 up to 256 takes, where its rings fit, the selected chain:
    "pair" (two steps per barrier, links eight cohorts back, P <= 64) or
    "prod"; otherwise K a
    multiple of 8 takes the producer-warp form (payload tiles: one, or two for
    K > 256), other K the per-thread-copy form.  Both launches (link pass and
    chain) are counted where the kernel applies; 512 members with 64-byte
    records and 128-byte payloads do not fit its rings and take the plain
    single-CTA kernel (one launch)."""
    import torch
    monkeypatch.setenv("RC_NO_PAIR", "0" if kernel == "pair" else "1")
    S = 256 if SB == 64 else 64
    N = K + extra
    tables, state0, outc, pay, idx = _inputs(90 + n_sets + K % 7, K, S, SB, P, n_sets, N=N)
    n = 70 if kernel == "pair" else 13  # the pair chain serves chains of 64 steps or more
    want = g.run_oracle(tables, state0, outc, pay, idx, n, sel0=1)
    got = g.run_gpu(rc.RC_MECH_RESIDENT_PERSIST, tables, state0, outc, pay, idx, n, K, sel0=1)
    g.assert_same(got, want, f"linked n_sets={n_sets} SB={SB} P={P} K={K} N={N}")
    ctx = rc.rc_init(S, tables, SB, P, K, N, torch.cuda.current_stream())
    try:
        state = g.dev(state0.copy())
        ev = rc.make_events(g.dev(outc), g.dev(pay), g.dev(idx), n_sets=n_sets)
        dec = torch.zeros(n, dtype=torch.int32, device="cuda")
        rc.rc_chain(ctx, n, rc.RC_MECH_RESIDENT_PERSIST, state, ev, K, dec)
        _, launches = rc.rc_last_chain_stats(ctx)
        assert launches == want_launches
    finally:
        rc.rc_free(ctx)


@pytest.mark.parametrize("cluster", [True, False])
@pytest.mark.parametrize("SB,P", [(16, 64), (64, 128), (16, 32)])
@pytest.mark.parametrize("K,extra,identity", [(513, 7, False), (1024, 0, False), (4100, 31, False), (8192, 5, False),
                                              (2048, 0, True)])
def test_cluster_chain(g, rc, monkeypatch, cluster, SB, P, K, extra, identity):
    """512 < K <= 8,192: one thread-block cluster (up to 16 CTAs) with the
    hardware cluster barrier, against the oracle; sessions drawn from K + extra
    so that most recur in the next step in another CTA of the cluster.  The
    grid kernels (cluster off) on the same inputs as a control."""
    monkeypatch.setenv("RC_NO_CLUSTER", "0" if cluster else "1")
    S = 256 if SB == 64 else 64
    tables, state0, outc, pay, idx = _inputs(110 + K % 13, K, S, SB, P, 5, N=None if identity else K + extra)
    n = 11
    want = g.run_oracle(tables, state0, outc, pay, idx, n, sel0=1)
    got = g.run_gpu(rc.RC_MECH_RESIDENT_PERSIST, tables, state0, outc, pay, idx, n, K, sel0=1)
    g.assert_same(got, want, f"cluster={cluster} K={K} SB={SB} P={P}")
