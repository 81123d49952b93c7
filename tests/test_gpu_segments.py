"""GPU parity of the segmented step (rc_seg_*: several route-keyed cohorts in
one launch, each route with its own pair of bodies and its own decision flag)
against the oracle's cohort step applied segment by segment with each
route's tables and flag.  Bit-exact on every decision, flag, effect and on
the final state."""
import importlib

import numpy as np
import pytest

import oracle
import rc_workload as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def g():
    return importlib.import_module("gpu_util")


@pytest.fixture(scope="module")
def rc():
    return importlib.import_module("paper_2608_12123_gb300")


def _route_tables(R, S, cfg):
    return np.stack([wl.make_tables(S, wl.stream_seed(cfg, wl.Purpose.TABLE, r)) for r in range(R)])


def _steps(R, N, P, T, cfg, sizes_hi, identity=False):
    """T steps: each a random subset of routes (in random order) with random
    segment sizes (0 allowed), sessions distinct across the step."""
    rng = np.random.default_rng(cfg)
    out = []
    for t in range(T):
        routes = rng.permutation(R)[: int(rng.integers(1, R + 1))].astype(np.uint32)
        sizes = rng.integers(0, sizes_hi + 1, len(routes))
        if t == 0:
            sizes[0] = 1
        total = int(sizes.sum())
        off = np.concatenate([[0], np.cumsum(sizes)]).astype(np.uint32)
        if identity:
            assert total <= N
            idx = None
        else:
            idx = wl.sample_without_replacement(N, total, wl.stream_seed(cfg, wl.Purpose.INDEX, t)).astype(np.uint32)
        outc, pay, _ = wl.make_cohort_events(cfg, 1, max(total, 1), P, set_offset=t)
        out.append((routes, off, outc[0][:total].copy(), pay[0][:total].copy(), idx))
    return out


def _oracle_steps(tables, state, steps, R):
    flags = np.zeros(R, dtype=np.uint32)
    res = []
    for routes, off, outc, pay, idx in steps:
        decs, effs = [], []
        for gi, r in enumerate(routes):
            a, b = int(off[gi]), int(off[gi + 1])
            # without an index array member m of the step (not of the segment) is session m
            seg_idx = np.arange(a, b, dtype=np.uint32) if idx is None else idx[a:b]
            d, eff, _ = oracle.cohort_step(tables[r], state, outc[a:b], pay[a:b], seg_idx, int(flags[r]))
            decs.append(d)
            effs.append(eff)
        for gi, r in enumerate(routes):
            flags[r] = decs[gi]
        res.append((np.array(decs, np.uint32), np.concatenate(effs) if effs else np.zeros((0, 16), np.uint8)))
    return res, flags


def _gpu_steps(g, rc, tables, state0, steps, R, S, SB, P, N):
    import torch
    max_members = max(int(off[-1]) for _, off, *_ in steps) + 1
    ctx = rc.rc_seg_init(R, S, tables, SB, P, max_members, R, N, torch.cuda.current_stream())
    try:
        state = g.dev(state0.copy())
        res = []
        for routes, off, outc, pay, idx in steps:
            total = int(off[-1])
            o = g.dev(outc if total else np.zeros(1, np.uint32))
            p = g.dev(pay if total else np.zeros((1, P), np.uint8))
            i = None if idx is None else g.dev(idx if total else np.zeros(1, np.uint32))
            ev = rc.make_events(o, p, i, payload_bytes=P, n_sets=1)
            dec = torch.zeros(len(routes), dtype=torch.int32, device="cuda")
            eff = torch.zeros(max(total, 1) * 16, dtype=torch.uint8, device="cuda")
            rc.rc_seg_step(ctx, state, ev, routes, off, dec, eff)
            rc.rc_seg_sync(ctx)
            res.append((g.host(dec, np.uint32).copy(), g.host(eff, np.uint8)[: total * 16].reshape(total, 16).copy()))
        flags = rc.rc_seg_get_flags(ctx)
        return res, flags, g.host(state, np.uint8).reshape(state0.shape)
    finally:
        rc.rc_seg_free(ctx)


@pytest.mark.parametrize("SB,P", [(16, 64), (64, 128), (16, 32), (64, 32)])
@pytest.mark.parametrize("R,N,hi", [(4, 3000, 400), (9, 20000, 1200), (2, 700, 300)])
def test_segmented_steps_match_the_oracle(g, rc, SB, P, R, N, hi):
    S = 256 if SB == 64 else 64
    cfg = 200 + R + SB + P
    tables = _route_tables(R, S, cfg)
    state0 = wl.make_state(N, S, SB, wl.stream_seed(cfg, wl.Purpose.STATE))
    steps = _steps(R, N, P, 12, cfg, hi)
    want_state = state0.copy()
    want, want_flags = _oracle_steps(tables, want_state, steps, R)
    got, got_flags, got_state = _gpu_steps(g, rc, tables, state0, steps, R, S, SB, P, N)
    for t, ((dw, ew), (dg, eg)) in enumerate(zip(want, got)):
        assert np.array_equal(dw, dg), f"step {t} decisions"
        assert np.array_equal(ew, eg), f"step {t} effects"
    assert np.array_equal(want_flags, got_flags)
    assert np.array_equal(want_state, got_state)
    assert 0 < sum(int(d.sum()) for d, _ in want) < sum(len(d) for d, _ in want)  # both bodies in play


def test_identity_sessions(g, rc):
    R, N, S, SB, P = 3, 900, 64, 16, 64
    tables = _route_tables(R, S, 301)
    state0 = wl.make_state(N, S, SB, wl.stream_seed(301, wl.Purpose.STATE))
    steps = _steps(R, N, P, 8, 301, 300, identity=True)
    want_state = state0.copy()
    want, want_flags = _oracle_steps(tables, want_state, steps, R)
    got, got_flags, got_state = _gpu_steps(g, rc, tables, state0, steps, R, S, SB, P, N)
    for (dw, ew), (dg, eg) in zip(want, got):
        assert np.array_equal(dw, dg) and np.array_equal(ew, eg)
    assert np.array_equal(want_flags, got_flags) and np.array_equal(want_state, got_state)


def test_layout_contract_and_latched_errors(g, rc):
    import torch
    R, N, S, SB, P = 3, 100, 16, 16, 32
    tables = _route_tables(R, S, 302)
    state0 = wl.make_state(N, S, SB, wl.stream_seed(302, wl.Purpose.STATE))
    ctx = rc.rc_seg_init(R, S, tables, SB, P, 64, R, N, torch.cuda.current_stream())
    try:
        state = g.dev(state0.copy())
        outc, pay, _ = wl.make_cohort_events(302, 1, 10, P)
        idx = np.arange(10, dtype=np.uint32)
        ev = rc.make_events(g.dev(outc[0]), g.dev(pay[0]), g.dev(idx), payload_bytes=P, n_sets=1)
        for routes, off in (([0, 0], [0, 5, 10]), ([0, 1], [0, 6, 5]), ([3], [0, 10]), ([0], [1, 10]),
                            ([0], [0, 65])):
            with pytest.raises(rc.RcError) as e:
                rc.rc_seg_step(ctx, state, ev, routes, off)
            assert e.value.code == rc.RC_E_INVAL
        bad = idx.copy()
        bad[7] = N
        ev2 = rc.make_events(g.dev(outc[0]), g.dev(pay[0]), g.dev(bad), payload_bytes=P, n_sets=1)
        rc.rc_seg_step(ctx, state, ev2, [1, 2], [0, 4, 10])
        with pytest.raises(rc.RcError) as e:
            rc.rc_seg_sync(ctx)
        assert e.value.code == rc.RC_E_INDEX
        # the context keeps working: a clean step right after
        rc.rc_seg_step(ctx, state, ev, [2], [0, 10])
        rc.rc_seg_sync(ctx)
    finally:
        rc.rc_seg_free(ctx)
