"""Pins for the fast-variant oracle (oracle/fast_ns.py, Sec. 4.3), CPU only.

The fixed-step iteration X <- X (a I + b X^T X + c (X^T X)^2) acts on singular values
only, so from X_0 = Delta / s it must equal U f(S / s) V^T with f the composed scalar
quintics; that identity is checked against LAPACK's SVD (numpy), independently of the
iteration.  Closed forms pin the scaling (c * orthogonal inputs) and the RMS proxy; the
LP's constraints and the interval chain pin the schedule.
"""
import os
import re

import numpy as np
import pytest

pytest.importorskip("scipy")
from oracle import fast_ns  # noqa: E402

COEFS5 = fast_ns.schedule(5)


def _rand(m, n, seed):
    return np.random.default_rng(seed).standard_normal((m, n))


@pytest.mark.parametrize("m,n", [(40, 24), (24, 40), (32, 32), (1, 7), (9, 1)])
def test_fixed_steps_act_on_singular_values_only(m, n):
    d = _rand(m, n, m * 31 + n)
    x, s = fast_ns.fast_polar(d, COEFS5)
    u, sv, vt = np.linalg.svd(d, full_matrices=False)
    assert s == pytest.approx(np.sqrt(np.sqrt(np.sum(sv ** 4))), rel=1e-13)   # ||D^T D||_F^(1/2)
    expect = (u * fast_ns.compose(COEFS5, sv / s)) @ vt
    assert np.linalg.norm(x - expect) <= 1e-12 * np.linalg.norm(expect)


def test_c_times_orthogonal_closed_form():
    q, _ = np.linalg.qr(_rand(50, 20, 3))
    c = 0.37
    u, sigma = fast_ns.fast_iso(c * q, COEFS5, alpha=2.0)
    assert sigma == pytest.approx(c, rel=1e-14)                      # RMS of equal singular values
    # s = ||(cQ)^T (cQ)||_F^(1/2) = c * 20^(1/4); every singular value of X_0 is 20^(-1/4)
    f = fast_ns.compose(COEFS5, np.array([20 ** -0.25]))[0]
    assert np.allclose(u, 2.0 * c * f * q, rtol=0, atol=1e-14)


def test_rms_proxy_dominates_the_mean_singular_value():
    d = _rand(30, 20, 5) @ np.diag(np.geomspace(1, 1e-3, 20))
    _, sigma = fast_ns.fast_iso(d, COEFS5)
    sv = np.linalg.svd(d, compute_uv=False)
    assert sigma == pytest.approx(np.sqrt(np.mean(sv ** 2)), rel=1e-13)
    assert sigma > sv.mean()


def test_fast_schedule_repeats_the_last_chain_step():
    sch = fast_ns.fast_schedule(10)
    assert sch[:7] == fast_ns.schedule(7) and sch[7:] == [sch[6]] * 3
    # the repeated step keeps values near 1 near 1 (no restart of the aggressive steps)
    y = fast_ns.compose(sch, np.geomspace(fast_ns.ELL, 1.0, 10001))
    assert np.abs(y - 1).max() < 2e-3


def test_zero_input():
    u, sigma = fast_ns.fast_iso(np.zeros((4, 3)), COEFS5)
    assert sigma == 0.0 and not u.any()


def test_schedule_constraints_and_interval_chain():
    lo, hi = fast_ns.ELL, fast_ns.HI
    errs = []
    for a, b, c in COEFS5:
        x = np.linspace(lo, hi, 200001)
        p = a * x + b * x ** 3 + c * x ** 5
        assert (p >= fast_ns.KAPPA * x - 1e-6).all()                 # the cushion holds
        errs.append(np.abs(1 - p).max())
        lo, hi = p.min() * (1 - fast_ns.GUARD), p.max() * (1 + fast_ns.GUARD)
    assert all(e2 < e1 for e1, e2 in zip(errs, errs[1:]))           # each step tightens the band
    # the composed map keeps every value of the design range inside the chain's own
    # prediction for the next step, which after 5 steps is within 15 % of 1
    y = fast_ns.compose(COEFS5, np.concatenate([np.geomspace(fast_ns.ELL, 1.0, 100001),
                                                np.linspace(fast_ns.ELL, fast_ns.HI, 100001)]))
    assert lo <= y.min() and y.max() <= hi
    assert 0.85 < lo and hi < 1.15


def test_compiled_schedule_matches_the_definition():
    """The library's compiled standard schedule is the same minimax chain (to LP accuracy)."""
    hdr = os.path.join(os.path.dirname(__file__), "..", "paper_2607_03011_gb300", "csrc", "ns_schedule.h")
    blk = open(hdr).read().split("static __constant__ float kSched[")[1].split("};")[0]
    compiled = [tuple(float(v) for v in r) for r in re.findall(r"\{([-0-9.e]+)f, ([-0-9.e]+)f, ([-0-9.e]+)f\}", blk)]
    mine = fast_ns.schedule(7)
    # the five steps the fast variant runs agree to the header's fp32 rounding; the last,
    # nearly flat step of the chain is less determined by the LP (different grids)
    for k, (a, b) in enumerate(zip(mine, compiled)):
        assert np.allclose(a, b, rtol=1e-6 if k < 5 else 1e-3, atol=0), (k, a, b)
    x = np.geomspace(1e-6, 1.0, 20001)
    f_mine, f_lib = fast_ns.compose(mine[:5], x), fast_ns.compose(compiled[:5], x)
    assert np.max(np.abs(f_mine - f_lib) / np.abs(f_lib)) < 1e-5


def test_outer_step_one_d_tensors_follow_nesterov():
    table = [(0, 4, 3), (12, 5, 0)]
    rng = np.random.default_rng(1)
    th, b, d = rng.standard_normal(17), rng.standard_normal(17), rng.standard_normal(17)
    out = fast_ns.isoloco_outer_step_fast(table, th, b, d, 1.0, 0.7, 0.9, COEFS5)
    nb = 0.9 * b[12:] + d[12:]
    assert np.allclose(out["momentum"][12:], nb) and np.allclose(out["theta"][12:], th[12:] - 0.7 * (d[12:] + 0.9 * nb))
    u, sigma = fast_ns.fast_iso(d[:12].reshape(4, 3), COEFS5)
    assert np.allclose(out["update"][:12], u.ravel()) and out["sigma_bar"][0] == pytest.approx(sigma)
    assert out["sigma_bar"][1] == 0.0
