"""Helpers for the GPU parity tests: run the CUDA path through the C ABI on
numpy inputs and compare every output with the CPU oracle."""
import numpy as np
import torch

import oracle
import paper_2608_12123_gb300 as rc


def dev(a):
    """numpy -> CUDA tensor with the same bytes (32-bit words as int32)."""
    if a is None:
        return None
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint32:
        a = a.view(np.int32)
    return torch.from_numpy(a).cuda()


def host(t, dtype):
    return t.cpu().numpy().view(dtype)


def run_gpu(mech, tables, state0, outc, pay, idx, n_steps, K, sel0=0, log=True, host_buffers=False,
            floor_seq=None, wait_ns=None):
    """One rc_chain on fresh copies of the inputs.  Returns a dict of numpy
    results (decisions, effects, state_log, state, sel)."""
    S = tables.shape[1]
    N, SB = state0.shape
    P = pay.shape[-1]
    ctx = rc.rc_init(S, tables, SB, P, max(K, 1), N, torch.cuda.current_stream())
    try:
        if wait_ns is not None:
            rc.rc_set_wait_limits(ctx, wait_ns, 60_000_000_000)
        if sel0:
            rc.rc_set_decision(ctx, sel0)
        state = dev(state0.copy())
        if host_buffers:
            o, p, i = np.ascontiguousarray(outc), np.ascontiguousarray(pay), (
                None if idx is None else np.ascontiguousarray(idx))
            dec = np.zeros(n_steps, np.uint32)
            eff = np.zeros((n_steps, K, 16), np.uint8) if log else None
            slog = np.zeros((n_steps, K, SB), np.uint8) if log else None
        else:
            o, p, i = dev(outc), dev(pay), dev(idx)
            dec = torch.zeros(max(n_steps, 1), dtype=torch.int32, device="cuda")
            eff = torch.zeros(max(n_steps * K * 16, 16), dtype=torch.uint8, device="cuda") if log else None
            slog = torch.zeros(max(n_steps * K * SB, 16), dtype=torch.uint8, device="cuda") if log else None
        n_sets = outc.shape[0] if outc.ndim == 2 else 1
        ev = rc.make_events(o, p, i, payload_bytes=P, n_sets=n_sets)
        if mech == rc.RC_MECH_FLOOR:
            seq = np.ascontiguousarray(floor_seq, dtype=np.uint32)
            rc.rc_chain(ctx, n_steps, mech, state, ev, K, seq, eff, slog)
            dec_np = seq
        else:
            rc.rc_chain(ctx, n_steps, mech, state, ev, K, dec, eff, slog)
            dec_np = dec if host_buffers else host(dec, np.uint32)[:n_steps]
        out = dict(decisions=np.asarray(dec_np)[:n_steps], state=host(state, np.uint8).reshape(N, SB),
                   sel=rc.rc_get_decision(ctx))
        if log:
            if host_buffers:
                out["effects"], out["state_log"] = eff, slog
            else:
                out["effects"] = host(eff, np.uint8)[:n_steps * K * 16].reshape(n_steps, K, 16)
                out["state_log"] = host(slog, np.uint8)[:n_steps * K * SB].reshape(n_steps, K, SB)
        return out
    finally:
        rc.rc_free(ctx)


def run_oracle(tables, state0, outc, pay, idx, n_steps, sel0=0, log=True):
    st = state0.copy()
    out = oracle.chain(tables, st, outc, pay, idx, n_steps, sel0=sel0, log=log)
    out["state"] = st
    return out


def first_diff(a, b):
    d = np.argwhere(np.asarray(a) != np.asarray(b))
    return None if len(d) == 0 else tuple(int(x) for x in d[0])


def assert_same(gpu, want, what=""):
    for k in ("decisions", "effects", "state_log", "state"):
        if k in gpu and want.get(k) is not None:
            g, w = np.asarray(gpu[k]), np.asarray(want[k])
            assert g.shape == w.shape, f"{what} {k}: shape {g.shape} != {w.shape}"
            assert np.array_equal(g, w), f"{what} {k}: first difference at {first_diff(g, w)}"
    if "sel" in want:
        assert gpu["sel"] == want["sel"], f"{what}: final flag {gpu['sel']} != {want['sel']}"
