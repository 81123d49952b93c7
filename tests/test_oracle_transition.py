"""Pins of the oracle's transition path (route key, state update, effect,
decision, chain) against values fixed outside the oracle: the published
SplitMix64 output vectors (tests/golden/splitmix64_kat.json), hand-worked
automaton tables, and invariants of a legal transition (Section 2.1: a
transition reads state and an event and emits new state, a route and an
effect; Section 7.1: one global binary decision per epoch selects the next
route body)."""
import json
import os

import numpy as np
import pytest

import oracle
import rc_workload as wl
from conftest import GOLDEN

M = (1 << 64) - 1
G = 0x9E3779B97F4A7C15
_KAT = json.load(open(os.path.join(GOLDEN, "splitmix64_kat.json")))
K0 = [int(x, 16) for x in _KAT["seed_0"]]
K1 = [int(x) for x in _KAT["seed_1234567"]]

# Hand-written automaton over S = 4 states and 8 outcome classes.
# T_A[1][3] = 2 while T_A[3][1] = 0, and T_B[1][3] = 1: a transposed index or a
# swapped body gives a different next state.
T_A = [[1, 0, 2, 3, 1, 0, 2, 3],
       [3, 2, 1, 2, 0, 1, 3, 2],
       [0, 1, 3, 2, 2, 3, 1, 0],
       [2, 0, 0, 1, 3, 2, 0, 1]]
T_B = [[3, 3, 1, 0, 2, 1, 0, 2],
       [1, 0, 2, 1, 3, 3, 1, 0],
       [2, 3, 0, 1, 1, 0, 2, 3],
       [0, 1, 3, 3, 0, 2, 1, 1]]
TABLES = np.array([T_A, T_B], dtype=np.uint8)


def le(w):
    return (w & M).to_bytes(8, "little")


def rotl(v, r):
    r %= 64
    return ((v << r) | (v >> (64 - r))) & M if r else v


def rec16(x, step, acc):
    return np.frombuffer(np.array([x], "<u4").tobytes() + np.array([step], "<u4").tobytes()
                         + np.array([acc], "<u8").tobytes(), dtype=np.uint8).copy()


def rec64(x, step, accs):
    b = np.array([x, step], "<u4").tobytes() + np.array(accs, "<u8").tobytes()
    return np.frombuffer(b, dtype=np.uint8).copy()


def fields16(rec):
    r = np.asarray(rec, dtype=np.uint8)
    return int(r[0:4].view("<u4")[0]), int(r[4:8].view("<u4")[0]), int(r[8:16].view("<u8")[0])


def effect_fields(e):
    e = np.asarray(e, dtype=np.uint8)
    return int(e[0:8].view("<u8")[0]), int(e[8:12].view("<u4")[0]), int(e[12:16].view("<u4")[0])


# ---------------------------------------------------------------- the mixer

def test_mix64_matches_published_splitmix64_vectors():
    for n, want in enumerate(K0, start=1):
        assert oracle.mix64((0 + n * G) & M) == want
    for n, want in enumerate(K1, start=1):
        assert oracle.mix64((1234567 + n * G) & M) == want


def test_input_generator_matches_published_vectors():
    assert [int(v) for v in wl.splitmix64(0, 4)] == K0
    assert [int(v) for v in wl.splitmix64(1234567, 5)] == K1
    # counter form: an offset continues the same stream
    assert [int(v) for v in wl.splitmix64(1234567, 2, offset=3)] == K1[3:5]


def test_mix64_is_a_bijection_on_a_sample():
    rng = np.random.default_rng(7)
    xs = {int(v) for v in rng.integers(0, 2**63, size=20000, dtype=np.int64)}
    ys = {oracle.mix64(x) for x in xs}
    assert len(ys) == len(xs)


# ------------------------------------------------------------- route key

def test_route_key_initial_round_and_word_chaining():
    # state 0, outcome 0, no payload: mix64(0 XOR gamma) = first output of seed 0
    assert oracle.route_key(0, 0, b"") == K0[0]
    # choose each little-endian payload word so the next round's input is
    # 1234567 + (k+1)*gamma: the k-th prefix must then give the k-th output
    h = K0[0]
    payload = b""
    for k in range(5):
        w = h ^ ((1234567 + (k + 1) * G) & M)
        payload += le(w)
        h = K1[k]
        assert oracle.route_key(0, 0, payload) == K1[k]
    # the same words read big-endian give a different key
    be = b"".join(payload[i:i + 8][::-1] for i in range(0, len(payload), 8))
    assert oracle.route_key(0, 0, be) != K1[4]


def test_route_key_packs_state_low_and_outcome_high():
    x = ((1234567 + G) & M) ^ G
    assert x < 2**32  # no carry crosses bit 32, so this is a pure state value
    assert oracle.route_key(x, 0, b"") == K1[0]
    # outcome sits at bit 32: the stream seeded so that seed + gamma hits
    # (3 | 5 << 32) XOR gamma must produce the key as its first output
    seed = (((3 | (5 << 32)) ^ G) - G) & M
    assert oracle.route_key(3, 5, b"") == int(wl.splitmix64(seed, 1)[0])
    assert oracle.route_key(3, 5, b"") != oracle.route_key(5, 3, b"")


# ----------------------------------------------------- one cohort step

def test_state_update_acc_step_and_pre_transition_key():
    for acc, want_acc in ((K0[0], 0), (K0[0] ^ 1, G), (K0[0] ^ 3, (3 * G) & M)):
        state = rec16(0, 7, acc)[None, :].copy()
        d, eff, ms = oracle.cohort_step(TABLES, state, np.array([0], np.uint32),
                                        np.zeros((1, 0), np.uint8), None, 0)
        x, step, a = fields16(state[0])
        # key from the state BEFORE the move (x = 0), although T_A[0][0] = 1
        assert effect_fields(eff[0]) == (K0[0], 0, 1)
        assert (x, step, a) == (1, 8, want_acc)
        assert d == 1  # one member, odd key
        assert bytes(ms[0]) == bytes(state[0])


def test_wide_record_rotates_key_by_8j_per_word():
    accs = [rotl(K0[0], 8 * j) ^ 1 for j in range(7)]
    state = rec64(0, 0, accs)[None, :].copy()
    oracle.cohort_step(TABLES, state, np.array([0], np.uint32), np.zeros((1, 0), np.uint8), None, 0)
    out = state[0, 8:64].view("<u8")
    assert [int(v) for v in out] == [G] * 7
    assert int(state[0, 4:8].view("<u4")[0]) == 1


def test_table_orientation_body_select_and_effect_packing():
    payload = np.arange(32, dtype=np.uint8).reshape(1, 32)
    for sel, want_y in ((0, T_A[1][3]), (1, T_B[1][3])):
        state = np.zeros((3, 16), np.uint8)
        state[2] = rec16(1, 0, 0)
        d, eff, ms = oracle.cohort_step(TABLES, state, np.array([3], np.uint32), payload,
                                        np.array([2], np.uint32), sel)
        rk, s, packed = effect_fields(eff[0])
        assert rk == oracle.route_key(1, 3, payload[0].tobytes())
        assert s == 2
        assert packed == want_y | (3 << 16) | (sel << 24)
        assert fields16(state[2])[0] == want_y
        assert not state[:2].any()  # other sessions untouched
    assert (T_A[1][3], T_B[1][3]) == (2, 1) and T_A[3][1] == 0
    assert 0x00030002 == T_A[1][3] | (3 << 16)
    assert 0x01030001 == T_B[1][3] | (3 << 16) | (1 << 24)


def _parity_cohort(parities):
    """Members on sessions with state 0, outcome 0 and one payload word
    chosen so the key is seed-0 output 3 (odd) or output 2 (even)."""
    K = len(parities)
    state = np.zeros((K, 16), np.uint8)
    words = [(K0[0] ^ ((3 if p else 2) * G)) & M for p in parities]
    payload = np.frombuffer(b"".join(le(w) for w in words), np.uint8).reshape(K, 8).copy()
    return state, np.zeros(K, np.uint32), payload


@pytest.mark.parametrize("parities,want", [
    ([1], 1), ([0], 0), ([1, 1, 0, 0], 0), ([1, 1, 1, 0], 1), ([0, 0, 0, 0], 0),
    ([1, 1, 0, 0, 0], 0), ([1, 1, 1, 0, 0], 1), ([1] * 7 + [0] * 7, 0), ([1] * 8 + [0] * 6, 1),
])
def test_decision_is_strict_majority_of_odd_keys(parities, want):
    state, outc, payload = _parity_cohort(parities)
    d, eff, _ = oracle.cohort_step(TABLES, state, outc, payload, None, 0)
    keys = [effect_fields(e)[0] for e in eff]
    assert keys == [K0[2] if p else K0[1] for p in parities]
    assert K0[2] & 1 == 1 and K0[1] & 1 == 0
    assert d == want


def test_empty_cohort_decides_zero():
    state = np.zeros((4, 16), np.uint8)
    d, eff, _ = oracle.cohort_step(TABLES, state, np.zeros(0, np.uint32), np.zeros((0, 8), np.uint8), None, 1)
    assert d == 0 and eff.shape == (0, 16) and not state.any()


def test_errors_out_of_range_state_outcome_index():
    state = np.zeros((2, 16), np.uint8)
    state[1] = rec16(4, 0, 0)  # 4 >= S
    with pytest.raises(oracle.OracleError) as e:
        oracle.cohort_step(TABLES, state, np.array([0], np.uint32), np.zeros((1, 8), np.uint8),
                           np.array([1], np.uint32), 0)
    assert e.value.code == oracle.E_STATE
    with pytest.raises(oracle.OracleError) as e:
        oracle.cohort_step(TABLES, np.zeros((2, 16), np.uint8), np.array([8], np.uint32),
                           np.zeros((1, 8), np.uint8), None, 0)
    assert e.value.code == oracle.E_STATE
    with pytest.raises(oracle.OracleError) as e:
        oracle.cohort_step(TABLES, np.zeros((2, 16), np.uint8), np.array([0], np.uint32),
                           np.zeros((1, 8), np.uint8), np.array([2], np.uint32), 0)
    assert e.value.code == oracle.E_INDEX


# ------------------------------------------------------------------ chain

def test_chain_decision_selects_next_body():
    state = rec16(0, 0, 0)[None, :].copy()
    outc = np.zeros((1, 1), np.uint32)
    pay = np.zeros((1, 1, 0), np.uint8)
    out = oracle.chain(TABLES, state, outc, pay, None, n_steps=2, sel0=0)
    # step 0: x = 0, key = K0[0] (odd) -> d0 = 1, y = T_A[0][0] = 1
    rk0, _, p0 = effect_fields(out["effects"][0, 0])
    assert (rk0, p0) == (K0[0], T_A[0][0])
    # step 1 runs body B because d0 = 1: y = T_B[1][0] = 1 (body A would give 3)
    _, _, p1 = effect_fields(out["effects"][1, 0])
    assert p1 == T_B[1][0] | (1 << 24)
    assert out["decisions"][0] == 1
    assert fields16(state[0])[1] == 2
    # a chain that starts on body B
    state = rec16(0, 0, 0)[None, :].copy()
    out = oracle.chain(TABLES, state, outc, pay, None, n_steps=1, sel0=1)
    assert effect_fields(out["effects"][0, 0])[2] == T_B[0][0] | (1 << 24)


def test_two_sessions_three_steps_worked_by_hand():
    """Two sessions over three chained steps of two members (S = 4, one
    payload word each, explicit session order changing between steps).
    Trajectory worked out by hand from T_A / T_B; each payload word is built
    from the hand-derived pre-step state so that the member's route key is a
    chosen published SplitMix64 output (seed 0, output k = mix(k * gamma)):
    the key matches only if the oracle enters the step with exactly that
    state, outcome and session.

    step 0, body A: s0 x=1 o=3 -> T_A[1][3]=2, key out 1 (odd); s1 x=3 o=1 ->
      T_A[3][1]=0, key out 3 (odd); 2 odd of 2 > 1 -> d0 = 1.
    step 1, body B: s1 x=0 o=2 -> T_B[0][2]=1 (A: 2), key out 2 (even); s0
      x=2 o=6 -> T_B[2][6]=2 (A: 1), key out 1 (odd); 1 odd -> d1 = 0.
    step 2, body A: s0 x=2 o=1 -> T_A[2][1]=1 (B: 3), key out 4 (even); s1
      x=1 o=4 -> T_A[1][4]=0 (B: 3), key out 3 (odd); 1 odd -> d2 = 0."""
    idx = np.array([[0, 1], [1, 0], [0, 1]], np.uint32)
    outc = np.array([[3, 1], [2, 6], [1, 4]], np.uint32)
    pre_x = [[1, 3], [0, 2], [2, 1]]   # hand-derived state entering each step
    out_k = [[1, 3], [2, 1], [4, 3]]   # published output chosen for each key
    post_x = [[2, 0], [1, 2], [1, 0]]  # hand-derived next states
    sels = [0, 1, 0]
    words = [[oracle.mix64((pre_x[j][m] | int(outc[j, m]) << 32) ^ G) ^ (out_k[j][m] * G & M)
              for m in range(2)] for j in range(3)]
    pay = np.frombuffer(b"".join(le(w) for row in words for w in row), np.uint8).reshape(3, 2, 8).copy()
    state = np.stack([rec16(1, 0, 0), rec16(3, 0, 0)])
    out = oracle.chain(TABLES, state, outc, pay, idx, n_steps=3, sel0=0)
    assert [int(d) for d in out["decisions"]] == [1, 0, 0]
    for j in range(3):
        for m in range(2):
            rk, s, packed = effect_fields(out["effects"][j, m])
            assert rk == K0[out_k[j][m] - 1], (j, m)
            assert s == idx[j, m]
            assert packed == post_x[j][m] | (int(outc[j, m]) << 16) | (sels[j] << 24), (j, m)
            x, step, _ = fields16(out["state_log"][j, m])
            assert (x, step) == (post_x[j][m], j + 1), (j, m)
    assert fields16(state[0])[:2] == (1, 3) and fields16(state[1])[:2] == (0, 3)
    assert out["sel"] == 0


def _random_chain(K=32, S=16, P=32, n_steps=200, SB=16, N=None, n_sets=7, cfg=91):
    tables = wl.make_tables(S, wl.stream_seed(cfg, wl.Purpose.TABLE))
    Nn = K if N is None else N
    state0 = wl.make_state(Nn, S, SB, wl.stream_seed(cfg, wl.Purpose.STATE))
    outc, pay, idx = wl.make_cohort_events(cfg, n_sets, K, P, n_sessions=N)
    return tables, state0, outc, pay, idx


@pytest.mark.parametrize("SB,N", [(16, None), (16, 200), (64, 100)])
def test_legal_transition_invariants_on_random_chain(SB, N):
    K, S, n_steps = 32, 16, 200
    tables, state0, outc, pay, idx = _random_chain(K=K, S=S, SB=SB, N=N, n_steps=n_steps)
    state = state0.copy()
    out = oracle.chain(tables, state, outc, pay, idx, n_steps=n_steps)
    n_sets = outc.shape[0]
    Nn = state.shape[0]
    visits = np.zeros(Nn, np.int64)
    cur = state0.copy()
    prev_d = 0
    for n in range(n_steps):
        j = n % n_sets
        members = np.arange(K) if idx is None else idx[j]
        odd = 0
        for m in range(K):
            s = int(members[m])
            rk, es, packed = effect_fields(out["effects"][n, m])
            y, o, sel = packed & 0xFFFF, (packed >> 16) & 0xFF, packed >> 24
            x_before = int(cur[s, 0:4].view("<u4")[0])
            assert es == s and o == outc[j, m] and sel == prev_d
            assert y < S and y == tables[sel, x_before, o]
            assert rk == oracle.route_key(x_before, o, pay[j, m].tobytes())
            rec = out["state_log"][n, m]
            assert int(rec[0:4].view("<u4")[0]) == y
            visits[s] += 1
            assert int(rec[4:8].view("<u4")[0]) == int(state0[s, 4:8].view("<u4")[0]) + visits[s]
            cur[s] = rec
            odd += rk & 1
        assert out["decisions"][n] == (1 if odd > K // 2 else 0)
        prev_d = int(out["decisions"][n])
    assert np.array_equal(cur, state)
    assert out["sel"] == prev_d


def test_chain_equals_repeated_single_steps():
    tables, state0, outc, pay, idx = _random_chain(K=16, S=8, SB=64, N=50, n_sets=3)
    a = state0.copy()
    out = oracle.chain(tables, a, outc, pay, idx, n_steps=9, sel0=1)
    b = state0.copy()
    sel = 1
    for n in range(9):
        j = n % 3
        d, eff, ms = oracle.cohort_step(tables, b, outc[j], pay[j], idx[j], sel)
        assert np.array_equal(eff, out["effects"][n]) and np.array_equal(ms, out["state_log"][n])
        assert d == out["decisions"][n]
        sel = d
    assert np.array_equal(a, b)
