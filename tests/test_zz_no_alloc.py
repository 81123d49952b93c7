"""rc_cohort_step_noalloc: the cohort step for callers that cannot allocate
device memory (their GPU memory belongs to another allocator, or they must not
allocate, and thereby synchronise, once serving).  It must give exactly what
rc_cohort_step gives, call after call, with nothing but the caller's buffers
and the library's fixed device scratch.  Kept in a file of its own, collected
last; it passes alone in a fresh process and after the other tests."""
import importlib

import numpy as np
import pytest

import rc_workload as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rc():
    return importlib.import_module("paper_2608_12123_gb300")


def _dev(a):
    import torch
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint32:
        a = a.view(np.int32)
    return torch.from_numpy(a).cuda()


@pytest.mark.parametrize("K,N,S,SB,P,sel0", [(300, 1000, 64, 16, 64, 0), (70_000, 100_000, 256, 64, 128, 1),
                                             (32, 32, 16, 16, 32, 1)])
def test_noalloc_step_matches_the_allocating_step_twice(rc, K, N, S, SB, P, sel0):
    import torch
    cfg = 900 + K % 97
    tables = wl.make_tables(S, wl.stream_seed(cfg, wl.Purpose.TABLE))
    state0 = wl.make_state(N, S, SB, wl.stream_seed(cfg, wl.Purpose.STATE))
    outc, pay, idx = wl.make_cohort_events(cfg, 2, K, P, n_sessions=N)
    stream = torch.cuda.current_stream()

    # reference: the allocating entry point, flag carried in its context
    ctx = rc.rc_init(S, tables, SB, P, K, N, stream)
    try:
        if sel0:
            rc.rc_set_decision(ctx, 1)
        st_a = _dev(state0.copy())
        eff_a, dec_a = [], []
        for j in range(2):
            e = torch.zeros(K * 16, dtype=torch.uint8, device="cuda")
            ev = rc.make_events(_dev(outc[j]), _dev(pay[j]), _dev(idx[j]), n_sets=1)
            rc.rc_cohort_step(ctx, st_a, ev, K, 0, e)
            dec_a.append(rc.rc_get_decision(ctx))
            eff_a.append(e.cpu().numpy())
        rc.rc_sync(ctx)
    finally:
        rc.rc_free(ctx)

    # the allocation-free entry point, flag and status in the caller's memory
    tab_d = _dev(tables.reshape(-1))
    flag = torch.full((1,), sel0, dtype=torch.int32, device="cuda")
    status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    st_b = _dev(state0.copy())
    for j in range(2):
        e = torch.zeros(K * 16, dtype=torch.uint8, device="cuda")
        ev = rc.make_events(_dev(outc[j]), _dev(pay[j]), _dev(idx[j]), n_sets=1)
        rc.rc_cohort_step_noalloc(tab_d, S, SB, P, st_b, N, ev, K, flag, e, status, stream)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        assert int(flag.item()) == dec_a[j], f"call {j}: decision"
        assert np.array_equal(e.cpu().numpy(), eff_a[j]), f"call {j}: effects"
    assert np.array_equal(st_b.cpu().numpy(), st_a.cpu().numpy()), "state after two calls"


def test_noalloc_rejects_a_cohort_beyond_its_scratch(rc):
    import torch
    K = 4096 * 256 + 8  # one CTA more than the fixed scratch holds
    tab_d = torch.zeros(2 * 16 * 8, dtype=torch.uint8, device="cuda")
    st = torch.zeros(16 * 16, dtype=torch.uint8, device="cuda")
    buf = torch.zeros(64, dtype=torch.int32, device="cuda")
    ev = rc.make_events(buf, torch.zeros(64 * 32, dtype=torch.uint8, device="cuda"), None, payload_bytes=32,
                        n_sets=1)
    flag = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(rc.RcError) as e:
        rc.rc_cohort_step_noalloc(tab_d, 16, 16, 32, st, 16, ev, K, flag)
    assert e.value.code == rc.RC_E_SIZE
    torch.cuda.synchronize()
    assert int(flag.item()) == 0  # nothing was launched
