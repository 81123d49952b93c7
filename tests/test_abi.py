"""The C ABI without a GPU: librc.so builds for sm_103a, loads, exports every
symbol include/rc.h declares with the constants the binding uses, and its
host-side cohort former (Section 9.1 online runtime; Eq. 1 feasibility)
matches the oracle's former cohort for cohort."""
import os
import re
import subprocess

import numpy as np
import pytest

from conftest import ROOT


def _builder():
    import importlib.util
    spec = importlib.util.spec_from_file_location("_rc_build", os.path.join(ROOT, "paper_2608_12123_gb300", "build.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


@pytest.fixture(scope="module")
def rc():
    _builder().build()
    import paper_2608_12123_gb300 as rc
    return rc


def _header():
    return open(os.path.join(ROOT, "include", "rc.h")).read()


def test_every_declared_symbol_is_exported(rc):
    declared = set(re.findall(r"^(?:int|int64_t|const char \*)\s*\*?(rc_[a-z_]+)\(", _header(), re.M))
    assert {"rc_init", "rc_cohort_step", "rc_chain", "rc_free"} <= declared
    out = subprocess.run(["nm", "-D", "--defined-only", rc.LIB_PATH], capture_output=True, text=True, check=True)
    exported = set(re.findall(r"\sT\s(rc_[a-z_]+)$", out.stdout, re.M))
    assert declared <= exported
    assert set(rc.EXPORTS) == declared
    for name in declared:
        assert hasattr(rc._lib, name)


def test_binding_constants_match_header(rc):
    h = _header()
    for name, val in re.findall(r"#define (RC_[A-Z_]+) \((-?\d+)\)", h) + re.findall(r"#define (RC_OK) (\d+)", h):
        assert getattr(rc, name) == int(val), name
    for name, val in re.findall(r"(RC_MECH_[A-Z_]+) = (\d+)", h):
        assert getattr(rc, name) == int(val), name


def test_library_is_built_for_sm_103a(rc):
    b = _builder()
    assert "arch=compute_103a,code=sm_103a" in b.ARCH


def test_rc_init_rejects_bad_arguments_without_touching_cuda(rc):
    tab = np.zeros((2, 16, 8), np.uint8)
    for args in [(15, np.zeros((2, 15, 8), np.uint8), 16, 32, 8, 8), (16, tab, 32, 32, 8, 8), (16, tab, 16, 48, 8, 8),
                 (16, tab, 16, 32, 0, 8), (16, tab, 16, 32, 8, 0)]:
        with pytest.raises(rc.RcError) as e:
            rc.rc_init(*args)
        assert e.value.code == rc.RC_E_INVAL
    bad = tab.copy()
    bad[1, 3, 5] = 16  # an entry >= S
    with pytest.raises(rc.RcError):
        rc.rc_init(16, bad, 16, 32, 8, 8)


@pytest.mark.parametrize("C,K,horizon", [(5000, 8, 10.0), (10000, 32, 10.0), (20000, 64, 20.0), (3000, 2, 5.0)])
def test_library_former_matches_oracle_former(rc, C, K, horizon):
    import oracle
    import rc_workload as wl
    panel = wl.make_panel()
    a = wl.make_arrivals(C, panel, horizon_s=horizon)
    m1, t1, r1 = rc.form_cohorts(a.t_ns, a.route, a.session, panel.n_labels, K, 50_000_000)
    m2, t2, r2 = oracle.former(a.t_ns, a.route, a.session, panel.n_labels, K, 50_000_000)
    assert m1.shape == m2.shape and len(m1) > 0
    assert np.array_equal(m1, m2) and np.array_equal(t1, t2) and np.array_equal(r1, r2)


def test_library_former_worked_fixture_and_counts(rc):
    import json
    from conftest import GOLDEN
    fx = json.load(open(os.path.join(GOLDEN, "former_worked.json")))
    f = rc.rc_former_create(fx["R"], fx["K"], fx["delta"])
    got = []
    for i, e in enumerate(fx["events"]):
        rc.rc_former_push(f, e["t"], e["route"], e["session"], i)
        while (c := rc.rc_former_pop(f)) is not None:
            got.append((c[0].tolist(), c[1]))
    assert [g[0] for g in got] == fx["cohorts"] and [g[1] for g in got] == fx["tau"]
    pushed, launched, fallback = rc.rc_former_counts(f)
    assert (pushed, launched, fallback) == (6, 4, 1)  # event 5 is still open
    rc.rc_former_free(f)


def test_library_former_rejects_disorder_and_bad_route(rc):
    f = rc.rc_former_create(2, 2, 10)
    rc.rc_former_push(f, 5, 0, 1, 0)
    with pytest.raises(rc.RcError):
        rc.rc_former_push(f, 4, 0, 2, 1)      # earlier time
    with pytest.raises(rc.RcError):
        rc.rc_former_push(f, 5, 0, 2, 0)      # same (t, id)
    with pytest.raises(rc.RcError):
        rc.rc_former_push(f, 6, 2, 2, 2)      # route out of range
    rc.rc_former_free(f)
