"""GB300-native ready-cohort transition engine (arXiv 2608.12123, "Ready Cohorts").

A ctypes binding of ``librc.so`` with the C ABI's names (``include/rc.h``):
``rc_init``, ``rc_cohort_step``, ``rc_chain``, ``rc_free`` and the helpers.
It marshals arguments only; every step of the path runs in the library's
CUDA kernels.  Buffers may be CUDA tensors (``torch``), host tensors or
numpy arrays; the library copies host buffers through device staging itself.

The library must be built first (``python paper_2608_12123_gb300/build.py`` or
``__graft_entry__.build()``).  There is no fallback: without ``librc.so`` the
import raises.
"""
from __future__ import annotations

import ctypes as C
import os

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_build", "librc.so")

RC_OK = 0
RC_E_INVAL = -1
RC_E_CUDA = -2
RC_E_DEADLINE = -3
RC_E_STATE = -4
RC_E_TIMEOUT = -5
RC_E_UNSUPPORTED = -6
RC_E_INDEX = -7
RC_E_NOMEM = -8
RC_E_SIZE = -9

RC_MECH_HOST_RT = 0
RC_MECH_RESIDENT_COND = 1
RC_MECH_RESIDENT_PERSIST = 2
RC_MECH_FIXED_NESTED = 3
RC_MECH_FLOOR = 4
RC_MECH_RESIDENT = 5

MECHANISMS = {"host_rt": RC_MECH_HOST_RT, "resident_cond": RC_MECH_RESIDENT_COND,
              "resident_persist": RC_MECH_RESIDENT_PERSIST, "fixed_nested": RC_MECH_FIXED_NESTED,
              "floor": RC_MECH_FLOOR, "resident": RC_MECH_RESIDENT}

#: every symbol include/rc.h declares
EXPORTS = ("rc_init", "rc_cohort_step", "rc_chain", "rc_free", "rc_last_error", "rc_sync",
           "rc_get_decision", "rc_set_decision", "rc_set_wait_limits", "rc_launch_floor",
           "rc_debug_skip_arrival", "rc_last_chain_stats", "rc_set_trace", "rc_cohort_step_noalloc", "rc_former_create", "rc_former_push", "rc_former_pop",
           "rc_former_push_many", "rc_former_pop_many", "rc_former_counts", "rc_former_free", "rc_opportunity",
           "rc_seg_init", "rc_seg_step", "rc_seg_sync", "rc_seg_get_flags", "rc_seg_set_flags", "rc_seg_last_error",
           "rc_seg_free", "rc_opportunity_grid")


class rc_opportunity_counts(C.Structure):
    _fields_ = [("n", C.c_uint64), ("fixed", C.c_uint64), ("exact", C.c_uint64), ("upper", C.c_uint64)]


class rc_events(C.Structure):
    _fields_ = [("outcome", C.c_void_p), ("payload", C.c_void_p), ("session_idx", C.c_void_p),
                ("payload_bytes", C.c_uint32), ("n_sets", C.c_uint32), ("launch_ns", C.c_int64)]


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with `python paper_2608_12123_gb300/build.py` "
                          "(there is no CPU fallback)")
    lib = C.CDLL(LIB_PATH)
    vp, u32, u64, i64, i = C.c_void_p, C.c_uint32, C.c_uint64, C.c_int64, C.c_int
    P = C.POINTER
    sig = {
        "rc_init": (i, [P(vp), u32, vp, u32, u32, u32, u64, vp]),
        "rc_cohort_step": (i, [vp, vp, P(rc_events), u32, i64, vp]),
        "rc_chain": (i, [vp, u32, i, vp, P(rc_events), u32, vp, vp, vp]),
        "rc_free": (i, [vp]),
        "rc_last_error": (C.c_char_p, [vp]),
        "rc_sync": (i, [vp]),
        "rc_get_decision": (i, [vp, P(u32)]),
        "rc_set_decision": (i, [vp, u32]),
        "rc_set_wait_limits": (i, [vp, u64, u64]),
        "rc_launch_floor": (i, [vp, i, u32, P(C.c_double)]),
        "rc_debug_skip_arrival": (i, [vp, u32]),
        "rc_last_chain_stats": (i, [vp, P(C.c_double), P(u32)]),
        "rc_set_trace": (i, [vp, vp, u64]),
        "rc_cohort_step_noalloc": (i, [vp, u32, u32, u32, vp, u64, P(rc_events), u32, vp, vp, vp, vp]),
        "rc_former_create": (i, [P(vp), u32, u32, i64]),
        "rc_former_push": (i, [vp, i64, u32, u32, i64]),
        "rc_former_pop": (i, [vp, vp, P(i64), P(u32)]),
        "rc_former_push_many": (i, [vp, u64, vp, vp, vp, i64]),
        "rc_former_pop_many": (i64, [vp, u64, vp, vp, vp]),
        "rc_former_counts": (i, [vp, P(i64), P(i64), P(i64)]),
        "rc_former_free": (i, [vp]),
        "rc_opportunity": (i, [vp, vp, u64, u32, u32, i64, i64, P(rc_opportunity_counts)]),
        "rc_seg_init": (i, [P(vp), u32, u32, vp, u32, u32, u32, u32, u64, vp]),
        "rc_seg_step": (i, [vp, vp, P(rc_events), u32, vp, vp, vp, vp]),
        "rc_seg_sync": (i, [vp]),
        "rc_seg_get_flags": (i, [vp, vp]),
        "rc_seg_set_flags": (i, [vp, vp]),
        "rc_seg_last_error": (C.c_char_p, [vp]),
        "rc_seg_free": (i, [vp]),
        "rc_opportunity_grid": (i, [vp, vp, u64, u32, vp, u32, vp, u32, i64, vp, vp]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    return lib


_lib = _load()


class RcError(RuntimeError):
    def __init__(self, code: int, message: str):
        super().__init__(f"rc error {code}: {message}")
        self.code = code


def _ptr(x):
    """Address of a buffer: torch tensor, numpy array, int or None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if hasattr(x, "ctypes"):
        return x.ctypes.data
    raise TypeError(f"not a buffer: {type(x)!r}")


class Ctx:
    """An rc_ctx* with the buffers it was given kept alive."""

    def __init__(self, handle):
        self.handle = handle

    def __bool__(self):
        return bool(self.handle)


def _check(ctx, rc):
    if rc != RC_OK:
        msg = _lib.rc_last_error(ctx.handle if isinstance(ctx, Ctx) else ctx)
        raise RcError(rc, msg.decode() if msg else "")
    return rc


def make_events(outcome, payload, session_idx=None, payload_bytes=None, n_sets=None, launch_ns=0):
    """Builds an rc_events from buffers holding n_sets cohorts (see rc.h)."""
    ev = rc_events()
    ev.outcome = _ptr(outcome)
    ev.payload = _ptr(payload)
    ev.session_idx = _ptr(session_idx)
    if payload_bytes is None:
        payload_bytes = int(payload.shape[-1])
    ev.payload_bytes = payload_bytes
    if n_sets is None:
        n_sets = int(outcome.shape[0]) if len(outcome.shape) == 2 else 1
    ev.n_sets = n_sets
    ev.launch_ns = int(launch_ns)
    ev._keep = (outcome, payload, session_idx)
    return ev


def rc_init(S, transition_table, state_bytes, payload_bytes, max_K, n_sessions, cuda_stream=None) -> Ctx:
    import numpy as np
    tab = np.ascontiguousarray(transition_table, dtype=np.uint8)
    if tab.size != 2 * S * 8:
        raise ValueError("transition_table must hold [2][S][8] bytes")
    h = C.c_void_p()
    stream = None
    if cuda_stream is not None:
        stream = cuda_stream if isinstance(cuda_stream, int) else int(cuda_stream.cuda_stream)
    rc = _lib.rc_init(C.byref(h), S, tab.ctypes.data, state_bytes, payload_bytes, max_K, n_sessions, stream)
    if rc != RC_OK:
        raise RcError(rc, "rc_init rejected its arguments or CUDA set-up failed")
    return Ctx(h)


def rc_cohort_step(ctx, state, events, K, deadline_ns, effects=None):
    return _check(ctx, _lib.rc_cohort_step(ctx.handle, _ptr(state), C.byref(events), K, int(deadline_ns),
                                           _ptr(effects)))


def rc_chain(ctx, n_steps, mechanism, state, events, K, decisions=None, effects=None, state_log=None):
    if isinstance(mechanism, str):
        mechanism = MECHANISMS[mechanism]
    return _check(ctx, _lib.rc_chain(ctx.handle, n_steps, mechanism, _ptr(state), C.byref(events), K,
                                     _ptr(decisions), _ptr(effects), _ptr(state_log)))


def rc_free(ctx):
    if ctx and ctx.handle:
        _lib.rc_free(ctx.handle)
        ctx.handle = None
    return RC_OK


def rc_last_error(ctx) -> str:
    msg = _lib.rc_last_error(ctx.handle)
    return msg.decode() if msg else ""


def rc_sync(ctx):
    return _check(ctx, _lib.rc_sync(ctx.handle))


def rc_get_decision(ctx) -> int:
    v = C.c_uint32()
    _check(ctx, _lib.rc_get_decision(ctx.handle, C.byref(v)))
    return int(v.value)


def rc_set_decision(ctx, sel):
    return _check(ctx, _lib.rc_set_decision(ctx.handle, sel))


def rc_set_wait_limits(ctx, device_ns, host_ns):
    return _check(ctx, _lib.rc_set_wait_limits(ctx.handle, int(device_ns), int(host_ns)))


def rc_launch_floor(ctx, kind, reps) -> float:
    v = C.c_double()
    _check(ctx, _lib.rc_launch_floor(ctx.handle, kind, reps, C.byref(v)))
    return float(v.value)


def rc_last_chain_stats(ctx):
    """(device milliseconds, kernel launches) of the last rc_chain's mechanism work."""
    ms = C.c_double()
    n = C.c_uint32()
    _check(ctx, _lib.rc_last_chain_stats(ctx.handle, C.byref(ms), C.byref(n)))
    return float(ms.value), int(n.value)


def rc_set_trace(ctx, buf, nbytes=None):
    """Points the profiling trace at a device buffer (None turns it off)."""
    if buf is None:
        return _check(ctx, _lib.rc_set_trace(ctx.handle, None, 0))
    if nbytes is None:
        nbytes = buf.numel() * buf.element_size()
    return _check(ctx, _lib.rc_set_trace(ctx.handle, _ptr(buf), int(nbytes)))


def rc_cohort_step_noalloc(tables, S, state_bytes, payload_bytes, state, n_sessions, events, K, flag,
                           effects=None, status=None, cuda_stream=None):
    """The allocation-free cohort step (see include/rc.h): every buffer is the
    caller's device memory; returns nothing, raises RcError on a rejected call."""
    stream = None
    if cuda_stream is not None:
        stream = cuda_stream if isinstance(cuda_stream, int) else int(cuda_stream.cuda_stream)
    rc = _lib.rc_cohort_step_noalloc(_ptr(tables), S, state_bytes, payload_bytes, _ptr(state), int(n_sessions),
                                     C.byref(events), K, _ptr(flag), _ptr(effects), _ptr(status), stream)
    if rc != RC_OK:
        raise RcError(rc, "rc_cohort_step_noalloc rejected the call" +
                      (" (K beyond its fixed scratch)" if rc == RC_E_SIZE else ""))


def rc_debug_skip_arrival(ctx, armed=True):
    return _check(ctx, _lib.rc_debug_skip_arrival(ctx.handle, 1 if armed else 0))


# ---- online cohort former -----------------------------------------------------

class Former:
    def __init__(self, handle, K):
        self.handle = handle
        self.K = K


def rc_former_create(n_routes, K, delta_ns) -> Former:
    h = C.c_void_p()
    rc = _lib.rc_former_create(C.byref(h), n_routes, K, int(delta_ns))
    if rc != RC_OK:
        raise RcError(rc, "rc_former_create rejected its arguments")
    return Former(h, K)


def rc_former_push(f, t_ns, route, session, event_id):
    rc = _lib.rc_former_push(f.handle, int(t_ns), int(route), int(session), int(event_id))
    if rc != RC_OK:
        raise RcError(rc, "rc_former_push: route out of range or event out of (t, id) order")


def rc_former_pop(f):
    """Returns (members int64 [K], tau, route) or None."""
    import numpy as np
    mem = np.zeros(f.K, dtype=np.int64)
    tau = C.c_int64()
    route = C.c_uint32()
    got = _lib.rc_former_pop(f.handle, mem.ctypes.data, C.byref(tau), C.byref(route))
    if got < 0:
        raise RcError(got, "rc_former_pop failed")
    return (mem, int(tau.value), int(route.value)) if got == 1 else None


def rc_former_counts(f):
    a, b, c = C.c_int64(), C.c_int64(), C.c_int64()
    _lib.rc_former_counts(f.handle, C.byref(a), C.byref(b), C.byref(c))
    return int(a.value), int(b.value), int(c.value)


def rc_former_free(f):
    if f and f.handle:
        _lib.rc_former_free(f.handle)
        f.handle = None


def form_cohorts(t_ns, route, session, n_routes, K, delta_ns):
    """Runs the library's former over events given in (t, id) order (id =
    position); returns (members int64 [nc][K], tau int64 [nc], route uint32 [nc])."""
    import numpy as np
    t_ns = np.ascontiguousarray(t_ns, dtype=np.int64)
    route = np.ascontiguousarray(route, dtype=np.uint32)
    session = np.ascontiguousarray(session, dtype=np.uint32)
    f = rc_former_create(n_routes, K, delta_ns)
    try:
        rc = _lib.rc_former_push_many(f.handle, len(t_ns), t_ns.ctypes.data, route.ctypes.data,
                                      session.ctypes.data, 0)
        if rc != RC_OK:
            raise RcError(rc, "rc_former_push_many rejected an event")
        cap = len(t_ns) // K + 1
        members = np.zeros((cap, K), dtype=np.int64)
        tau = np.zeros(cap, dtype=np.int64)
        rr = np.zeros(cap, dtype=np.uint32)
        nc = _lib.rc_former_pop_many(f.handle, cap, members.ctypes.data, tau.ctypes.data, rr.ctypes.data)
        if nc < 0:
            raise RcError(int(nc), "rc_former_pop_many failed")
        return members[:nc], tau[:nc], rr[:nc]
    finally:
        rc_former_free(f)


def rc_opportunity(t_ns, route, n_routes, K, delta_ns, origin_ns=0):
    """Counts {n, fixed, exact, upper}: the events that fixed windows (F, Eq. 2),
    the exact offline packing (P*, Eq. 6) and the upper bound (U, Eqs. 3-4)
    serve at threshold K and deadline delta_ns."""
    import numpy as np
    t_ns = np.ascontiguousarray(t_ns, dtype=np.int64)
    route = np.ascontiguousarray(route, dtype=np.uint32)
    out = rc_opportunity_counts()
    rc = _lib.rc_opportunity(t_ns.ctypes.data, route.ctypes.data, len(t_ns), n_routes, K, delta_ns, origin_ns,
                             C.byref(out))
    if rc != RC_OK:
        raise RcError(rc, "rc_opportunity rejected its arguments")
    return dict(n=int(out.n), fixed=int(out.fixed), exact=int(out.exact), upper=int(out.upper))


def opportunity_shares(t_ns, route, n_routes, K, delta_ns, launched, origin_ns=0):
    """F, P*, U and A as fractions of the events, G (Eq. 7) and R_A (Eq. 9)
    from rc_opportunity and the former's launched-event count."""
    c = rc_opportunity(t_ns, route, n_routes, K, delta_ns, origin_ns)
    n, f, p, u = c["n"], c["fixed"], c["exact"], c["upper"]
    out = dict(n=n, F=f / n if n else 0.0, P=p / n if n else 0.0, U=u / n if n else 0.0,
               A=launched / n if n else 0.0, counts=dict(F=f, P=p, U=u, A=int(launched)))
    out["G"] = (p - f) / (u - f) if u > f else None
    out["R_A"] = (launched - f) / (p - f) if p > f else None
    return out


class SegCtx:
    """A segmented-step context (rc_seg_*): n_routes routes, each with its own
    pair of bodies and its own device-resident flag."""

    def __init__(self, handle, n_routes):
        self.handle = handle
        self.n_routes = n_routes


def _seg_check(ctx, rc):
    if rc != RC_OK:
        msg = _lib.rc_seg_last_error(ctx.handle) if ctx and ctx.handle else b""
        raise RcError(rc, msg.decode() if msg else "")


def rc_seg_init(n_routes, S, tables, state_bytes, payload_bytes, max_members, max_segments, n_sessions, stream=None):
    """tables: uint8 [n_routes][2][S][8] (body A then B per route)."""
    import numpy as np
    tables = np.ascontiguousarray(tables, dtype=np.uint8)
    if tables.size != n_routes * 2 * S * 8:
        raise ValueError("tables must hold n_routes x 2 x S x 8 entries")
    h = C.c_void_p()
    st = None if stream is None else (stream if isinstance(stream, int) else int(stream.cuda_stream))
    rc = _lib.rc_seg_init(C.byref(h), n_routes, S, tables.ctypes.data, state_bytes, payload_bytes, max_members,
                          max_segments, n_sessions, st)
    if rc != RC_OK:
        raise RcError(rc, "rc_seg_init failed")
    return SegCtx(h.value, n_routes)


def rc_seg_step(ctx, state, events, seg_route, seg_off, decisions=None, effects=None):
    """seg_route, seg_off: host integer arrays (n and n + 1 entries)."""
    import numpy as np
    seg_route = np.ascontiguousarray(seg_route, dtype=np.uint32)
    seg_off = np.ascontiguousarray(seg_off, dtype=np.uint32)
    if len(seg_off) != len(seg_route) + 1:
        raise ValueError("seg_off needs one entry more than seg_route")
    _seg_check(ctx, _lib.rc_seg_step(ctx.handle, _ptr(state), C.byref(events), len(seg_route), seg_route.ctypes.data,
                                     seg_off.ctypes.data, _ptr(decisions), _ptr(effects)))


def rc_seg_sync(ctx):
    _seg_check(ctx, _lib.rc_seg_sync(ctx.handle))


def rc_seg_get_flags(ctx):
    import numpy as np
    out = np.zeros(ctx.n_routes, dtype=np.uint32)
    _seg_check(ctx, _lib.rc_seg_get_flags(ctx.handle, out.ctypes.data))
    return out


def rc_seg_set_flags(ctx, flags):
    import numpy as np
    flags = np.ascontiguousarray(flags, dtype=np.uint32)
    _seg_check(ctx, _lib.rc_seg_set_flags(ctx.handle, flags.ctypes.data))


def rc_seg_free(ctx):
    if ctx and ctx.handle:
        _lib.rc_seg_free(ctx.handle)
        ctx.handle = None


def rc_opportunity_grid(t_ns, route, n_routes, K_list, delta_list, origin_ns=0, stream=None):
    """{fixed, exact, upper} for every (delta, K) pair, on the GPU: returns a
    uint64 array [len(delta_list)][len(K_list)][3]."""
    import numpy as np
    t_ns = np.ascontiguousarray(t_ns, dtype=np.int64)
    route = np.ascontiguousarray(route, dtype=np.uint32)
    ks = np.ascontiguousarray(K_list, dtype=np.uint32)
    ds = np.ascontiguousarray(delta_list, dtype=np.int64)
    out = np.zeros((len(ds), len(ks), 3), dtype=np.uint64)
    st = None if stream is None else (stream if isinstance(stream, int) else int(stream.cuda_stream))
    rc = _lib.rc_opportunity_grid(t_ns.ctypes.data, route.ctypes.data, len(t_ns), n_routes, ks.ctypes.data, len(ks),
                                  ds.ctypes.data, len(ds), origin_ns, out.ctypes.data, st)
    if rc != RC_OK:
        raise RcError(rc, "rc_opportunity_grid failed")
    return out
