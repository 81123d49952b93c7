"""CPU oracle for the ready-cohort transition path (test infrastructure).

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  It wraps ``rc_oracle.c`` (plain C,
single-threaded) through ctypes and shares no code with the CUDA path; inputs
come from :mod:`rc_workload`.

What each function computes, and the passage it follows, is stated in
``rc_oracle.c``.  Pins: every function here is checked in ``tests/`` against
published SplitMix64 vectors, brute force on tiny inputs, closed forms and the
paper's invariants (Proposition 1 and the five validity gates of Section 5.3).
The paper's own trace figures are not reproduced (parity unpinned for those
numbers: the trace panel is not available).
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "rc_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

OK = 0
E_INVAL = -1
E_STATE = -4
E_INDEX = -7


def build(force: bool = False) -> str:
    """Compile rc_oracle.c into _build/liboracle.so (gcc, -O2, C11)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    fresh = os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)
    if force or not fresh:
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.run(["gcc", "-O2", "-std=c11", "-Wall", "-Wextra", "-fPIC", "-shared",
                        _SRC, "-o", tmp], check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = C.CDLL(build())
        u8p, u32p, i64p = C.POINTER(C.c_uint8), C.POINTER(C.c_uint32), C.POINTER(C.c_int64)
        lib.orc_mix64.restype = C.c_uint64
        lib.orc_mix64.argtypes = [C.c_uint64]
        lib.orc_route_key.restype = C.c_uint64
        lib.orc_route_key.argtypes = [C.c_uint32, C.c_uint32, u8p, C.c_uint32]
        lib.orc_cohort_step.restype = C.c_int
        lib.orc_cohort_step.argtypes = [C.c_uint32, u8p, C.c_uint32, u8p, C.c_uint64, u32p, u8p,
                                        C.c_uint32, u32p, C.c_uint32, C.c_uint32, u8p, u8p, u32p]
        lib.orc_chain.restype = C.c_int
        lib.orc_chain.argtypes = [C.c_uint32, u8p, C.c_uint32, u8p, C.c_uint64, u32p, u8p, C.c_uint32,
                                  u32p, C.c_uint32, C.c_uint32, C.c_uint32, C.c_uint32, u32p, u8p, u8p, u32p]
        lib.orc_fixed_count.restype = C.c_int64
        lib.orc_fixed_count.argtypes = [C.c_int64, i64p, u32p, C.c_uint32, u32p, C.c_int64, C.c_int64]
        lib.orc_upper_count.restype = C.c_int64
        lib.orc_upper_count.argtypes = [C.c_int64, i64p, u32p, C.c_uint32, u32p, C.c_int64, u8p]
        lib.orc_exact_count.restype = C.c_int64
        lib.orc_exact_count.argtypes = [C.c_int64, i64p, u32p, C.c_uint32, u32p, C.c_int64, C.c_int,
                                        i64p, i64p]
        lib.orc_former.restype = C.c_int64
        lib.orc_former.argtypes = [C.c_int64, i64p, u32p, u32p, C.c_uint32, C.c_uint32, C.c_int64,
                                   i64p, i64p, u32p, C.c_int64]
        _lib = lib
        return lib


def _p(a, ctype):
    if a is None:
        return None
    return a.ctypes.data_as(C.POINTER(ctype))


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


class OracleError(RuntimeError):
    def __init__(self, code):
        super().__init__(f"oracle error {code}")
        self.code = code


def mix64(z: int) -> int:
    return int(_load().orc_mix64(z & ((1 << 64) - 1)))


def route_key(x: int, o: int, payload: bytes | np.ndarray) -> int:
    p = _c(np.frombuffer(bytes(payload), dtype=np.uint8) if isinstance(payload, (bytes, bytearray))
           else payload, np.uint8)
    return int(_load().orc_route_key(x, o, _p(p, C.c_uint8), len(p)))


def cohort_step(tables, state, outcome, payload, idx, sel):
    """One cohort step on ``state`` (uint8 [N][SB], updated in place).
    Returns (d, effects uint8 [K][16], member_state uint8 [K][SB])."""
    lib = _load()
    tables = _c(tables, np.uint8)
    S = tables.shape[1]
    assert state.flags.c_contiguous and state.dtype == np.uint8
    N, SB = state.shape
    outcome = _c(outcome, np.uint32)
    K = outcome.shape[0]
    payload = _c(payload, np.uint8)
    if payload.ndim != 2:
        payload = payload.reshape(K, -1)
    P = payload.shape[1]
    idx = None if idx is None else _c(idx, np.uint32)
    eff = np.zeros((K, 16), dtype=np.uint8)
    ms = np.zeros((K, SB), dtype=np.uint8)
    d = np.zeros(1, dtype=np.uint32)
    rc = lib.orc_cohort_step(S, _p(tables, C.c_uint8), SB, _p(state, C.c_uint8), N, _p(outcome, C.c_uint32),
                             _p(payload, C.c_uint8), P, _p(idx, C.c_uint32), K, sel,
                             _p(eff, C.c_uint8), _p(ms, C.c_uint8), _p(d, C.c_uint32))
    if rc != OK:
        raise OracleError(rc)
    return int(d[0]), eff, ms


def chain(tables, state, outcome, payload, idx, n_steps, sel0=0, log=True):
    """A chain of n_steps cohort steps over event sets outcome [n_sets][K],
    payload [n_sets][K][P], idx [n_sets][K] or None; step n uses set n mod
    n_sets.  ``state`` (uint8 [N][SB]) is updated in place.  Returns a dict
    with decisions [n_steps], effects [n_steps][K][16] and state_log
    [n_steps][K][SB] (when log), and the final sel."""
    lib = _load()
    tables = _c(tables, np.uint8)
    S = tables.shape[1]
    assert state.flags.c_contiguous and state.dtype == np.uint8
    N, SB = state.shape
    outcome = _c(outcome, np.uint32)
    if outcome.ndim == 1:
        outcome = outcome[None]
    n_sets, K = outcome.shape
    payload = _c(payload, np.uint8).reshape(n_sets, K, -1)
    P = payload.shape[2]
    idx = None if idx is None else _c(idx, np.uint32).reshape(n_sets, K)
    dec = np.zeros(n_steps, dtype=np.uint32)
    eff = np.zeros((n_steps, K, 16), dtype=np.uint8) if log else None
    slog = np.zeros((n_steps, K, SB), dtype=np.uint8) if log else None
    sel = np.zeros(1, dtype=np.uint32)
    rc = lib.orc_chain(S, _p(tables, C.c_uint8), SB, _p(state, C.c_uint8), N, _p(outcome, C.c_uint32),
                       _p(payload, C.c_uint8), P, _p(idx, C.c_uint32), n_sets, K, n_steps, sel0,
                       _p(dec, C.c_uint32), _p(eff, C.c_uint8), _p(slog, C.c_uint8), _p(sel, C.c_uint32))
    if rc != OK:
        raise OracleError(rc)
    return dict(decisions=dec, effects=eff, state_log=slog, sel=int(sel[0]))


def _kr(Kr, R):
    if np.isscalar(Kr):
        return np.full(R, int(Kr), dtype=np.uint32)
    return _c(Kr, np.uint32)


def fixed_count(t, route, R, Kr, delta, origin=0) -> int:
    """Eq. 2 numerator: events in (window, route) buckets with n_b >= K_r."""
    t = _c(t, np.int64)
    route = _c(route, np.uint32)
    kr = _kr(Kr, R)
    v = _load().orc_fixed_count(len(t), _p(t, C.c_int64), _p(route, C.c_uint32), R, _p(kr, C.c_uint32),
                                delta, origin)
    if v < 0:
        raise OracleError(v)
    return int(v)


def upper_count(t, route, R, Kr, delta, want_eligible=False):
    """Eq. 4 numerator (and the per-event indicator when asked)."""
    t = _c(t, np.int64)
    route = _c(route, np.uint32)
    kr = _kr(Kr, R)
    el = np.zeros(len(t), dtype=np.uint8) if want_eligible else None
    v = _load().orc_upper_count(len(t), _p(t, C.c_int64), _p(route, C.c_uint32), R, _p(kr, C.c_uint32),
                                delta, _p(el, C.c_uint8))
    if v < 0:
        raise OracleError(v)
    return (int(v), el) if want_eligible else int(v)


def exact_count(t, route, R, Kr, delta, method=0, want_witness=False):
    """Maximum number of events assigned in a feasible offline schedule
    (P* numerator).  method 0 = Algorithm 1 (monotone deque, with witness),
    method 1 = Eq. 6 scanned directly."""
    t = _c(t, np.int64)
    route = _c(route, np.uint32)
    kr = _kr(Kr, R)
    bo = np.zeros(len(t), dtype=np.int64) if want_witness else None
    nb = np.zeros(1, dtype=np.int64)
    v = _load().orc_exact_count(len(t), _p(t, C.c_int64), _p(route, C.c_uint32), R, _p(kr, C.c_uint32),
                                delta, method, _p(bo, C.c_int64), _p(nb, C.c_int64))
    if v < 0:
        raise OracleError(v)
    return (int(v), bo, int(nb[0])) if want_witness else int(v)


def former(t, route, session, R, K, delta, cap=None):
    """Online cohort former.  Returns (members int64 [nc][K] event ids,
    tau int64 [nc], croute uint32 [nc]) for the cohorts in launch order."""
    lib = _load()
    t = _c(t, np.int64)
    route = _c(route, np.uint32)
    session = _c(session, np.uint32)
    n = len(t)
    if cap is None:
        cap = n // max(K, 1) + 1
    mem = np.zeros((cap, K), dtype=np.int64)
    tau = np.zeros(cap, dtype=np.int64)
    cr = np.zeros(cap, dtype=np.uint32)
    nc = lib.orc_former(n, _p(t, C.c_int64), _p(route, C.c_uint32), _p(session, C.c_uint32), R, K, delta,
                        _p(mem, C.c_int64), _p(tau, C.c_int64), _p(cr, C.c_uint32), cap)
    if nc < 0:
        raise OracleError(nc)
    k = min(nc, cap)
    return mem[:k], tau[:k], cr[:k]


def shares(t, route, session, R, K, delta, origin=0):
    """F, P*, U (Eqs. 2, 4 and Section 4) and the former's A, as fractions of
    |E|, plus G (Eq. 7) and R_A (Eq. 9) where their denominators are positive."""
    n = len(t)
    f = fixed_count(t, route, R, K, delta, origin)
    p = exact_count(t, route, R, K, delta)
    u = upper_count(t, route, R, K, delta)
    mem, _, _ = former(t, route, session, R, K, delta)
    a = mem.size
    out = dict(n=n, F=f / n if n else 0.0, P=p / n if n else 0.0, U=u / n if n else 0.0,
               A=a / n if n else 0.0, counts=dict(F=f, P=p, U=u, A=a))
    out["G"] = (p - f) / (u - f) if u > f else None
    out["R_A"] = (a - f) / (p - f) if p > f else None
    return out
