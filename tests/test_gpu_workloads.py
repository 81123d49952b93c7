"""GPU parity on the five workload shapes at their full sizes (bit-exact on
every decision, effect and state field; Sections 2.2 and 7.3):

  tiny chain       K=32, S=16, 1,000 steps (also in test_gpu_parity)
  cohort replay    cohorts formed from Poisson arrivals for C=100,000, K=256
  sweep cells      C in {10k, 100k} x K in {32, 64, 128, 256}, three mechanisms
  large cohort     N=1,048,576 64-byte records, K=65,536, 128-byte payloads,
                   S=256, the 1,000-invocation launch the benchmark times
  long chain       K=256, S=128, 10,000 steps, 50 seeds, resident and host RT
"""
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


@pytest.fixture(scope="module")
def panel():
    return wl.make_panel()


def _formed(rc, panel, C, K, delta=50_000_000):
    a = wl.make_arrivals(C, panel)
    mem, tau, cr = rc.form_cohorts(a.t_ns, a.route, a.session, panel.n_labels, K, delta)
    return a, mem, tau, cr


def _cohort_inputs(a, mem, P=64, S=64, cfg=2):
    K = mem.shape[1]
    outc = (a.route[mem] % 8).astype(np.uint32)
    idx = a.session[mem].astype(np.uint32)
    pay = wl.payload_for_events(mem.reshape(-1), P).reshape(len(mem), K, P)
    tables = wl.make_tables(S, wl.stream_seed(cfg, wl.Purpose.TABLE))
    state0 = wl.make_state(a.n_sessions, S, 16, wl.stream_seed(cfg, wl.Purpose.STATE))
    return tables, state0, outc, pay, idx


@pytest.fixture(scope="module")
def replay(rc, panel):
    a, mem, tau, cr = _formed(rc, panel, 100_000, 256)
    # the library's former and the oracle's agree on the full replay
    m2, t2, r2 = oracle.former(a.t_ns, a.route, a.session, panel.n_labels, 256, 50_000_000)
    assert np.array_equal(mem, m2) and np.array_equal(tau, t2) and np.array_equal(cr, r2)
    return a, mem


def test_replay_first_1000_cohorts_every_mechanism(g, rc, replay):
    a, mem = replay
    n = 1000
    tables, state0, outc, pay, idx = _cohort_inputs(a, mem[:n])
    want = g.run_oracle(tables, state0, outc, pay, idx, n)
    for name in ("resident_persist", "host_rt", "resident_cond", "fixed_nested", "floor"):
        got = g.run_gpu(rc.MECHANISMS[name], tables, state0, outc, pay, idx, n, 256, floor_seq=want["decisions"])
        w = dict(want)
        if name == "floor":
            w.pop("sel")
        g.assert_same(got, w, f"replay {name}")


def test_replay_all_cohorts_resident(g, rc, replay):
    a, mem = replay
    n = len(mem)
    tables, state0, outc, pay, idx = _cohort_inputs(a, mem)
    want = g.run_oracle(tables, state0, outc, pay, idx, n, log=False)
    got = g.run_gpu(rc.RC_MECH_RESIDENT, tables, state0, outc, pay, idx, n, 256, log=False)
    g.assert_same(got, want, "replay, all cohorts")
    assert 0 < want["decisions"].sum() < n


@pytest.mark.parametrize("C", [10_000, 100_000])
@pytest.mark.parametrize("K", [32, 64, 128, 256])
def test_sweep_cells(g, rc, panel, C, K):
    a, mem, tau, cr = _formed(rc, panel, C, K)
    if len(mem) == 0:
        # no qualifying cohort in this cell (the paper reports such cells too)
        assert K >= 64 and C == 10_000
        return
    n = min(1000, len(mem))
    tables, state0, outc, pay, idx = _cohort_inputs(a, mem[:n])
    want = g.run_oracle(tables, state0, outc, pay, idx, n, log=False)
    for name in ("host_rt", "resident_persist", "fixed_nested", "resident_cond"):
        got = g.run_gpu(rc.MECHANISMS[name], tables, state0, outc, pay, idx, n, K, log=False)
        g.assert_same(got, want, f"C={C} K={K} {name}")


@pytest.fixture(scope="module")
def large():
    c = wl.CONFIGS[4]
    tables = wl.make_tables(c["S"], wl.stream_seed(4, wl.Purpose.TABLE))
    state0 = wl.make_state(c["N"], c["S"], c["state_bytes"], wl.stream_seed(4, wl.Purpose.STATE))
    outc, pay, idx = wl.make_cohort_events(4, c["n_sets"], c["K"], c["payload_bytes"], n_sessions=c["N"])
    return tables, state0, outc, pay, idx


def test_large_cohort_logged_steps_every_mechanism(g, rc, large):
    tables, state0, outc, pay, idx = large
    K, n = 65_536, 12
    want = g.run_oracle(tables, state0, outc[:8], pay[:8], idx[:8], n)
    for name in ("resident_persist", "host_rt", "resident_cond"):
        got = g.run_gpu(rc.MECHANISMS[name], tables, state0, outc[:8], pay[:8], idx[:8], n, K)
        g.assert_same(got, want, f"large K {name}")


def test_large_cohort_benchmark_launch(g, rc, large):
    """The 1,000-invocation resident chain over the 64-set ring, as timed."""
    tables, state0, outc, pay, idx = large
    K, n = 65_536, 1000
    want = g.run_oracle(tables, state0, outc, pay, idx, n, log=False)
    got = g.run_gpu(rc.RC_MECH_RESIDENT, tables, state0, outc, pay, idx, n, K, log=False)
    g.assert_same(got, want, "large K, 1,000 invocations")


def _stress_inputs(seed):
    c = wl.CONFIGS[5]
    cfg = 1000 + seed
    tables = wl.make_tables(c["S"], wl.stream_seed(cfg, wl.Purpose.TABLE))
    state0 = wl.make_state(c["K"], c["S"], 16, wl.stream_seed(cfg, wl.Purpose.STATE))
    outc, pay, _ = wl.make_cohort_events(cfg, c["n_steps"], c["K"], c["payload_bytes"])
    return tables, state0, outc, pay


@pytest.mark.parametrize("block", range(5))
def test_long_chain_fifty_seeds(g, rc, block):
    """K=256, S=128, 10,000 steps, A/B tables; 10 seeds per block, 50 in all;
    every step's states, effects and decision compared."""
    n = wl.CONFIGS[5]["n_steps"]
    for seed in range(10 * block, 10 * block + 10):
        tables, state0, outc, pay = _stress_inputs(seed)
        want = g.run_oracle(tables, state0, outc, pay, None, n)
        assert 0 < want["decisions"].sum() < n
        for name in ("resident_persist", "host_rt"):
            got = g.run_gpu(rc.MECHANISMS[name], tables, state0, outc, pay, None, n, 256)
            g.assert_same(got, want, f"seed {seed} {name}")
