"""Pins for the ablation oracle (oracle/variants.py, Sec. 4.5 and App. B), CPU only.

Each variant is pinned by what does not depend on the oracle's own sequencing: the
default flags reproduce the pinned Alg. 2 oracle, mu = 0 collapses every momentum choice
to Eq. 2 (plain SGD on the Iso-C direction), inputs that are c * orthogonal (with momentum
along the same direction) have closed forms for every variant, and a scalar worked by
hand pins standard momentum.
"""
import numpy as np
import pytest

import oracle
from oracle import variants

TABLE = [(0, 6, 4), (24, 3, 5), (39, 5, 0)]     # two matrices and a vector
N = 44


def _inputs(seed, k=3):
    rng = np.random.default_rng(seed)
    theta = (0.02 * rng.standard_normal(N)).astype(np.float32)
    reps = [(theta - 1e-3 * rng.standard_normal(N)).astype(np.float32) for _ in range(k)]
    mom = (1e-3 * rng.standard_normal(N)).astype(np.float32)
    return theta, mom, np.stack(reps)


def test_default_flags_reproduce_alg2():
    th, b, reps = _inputs(1)
    ref = oracle.isoloco_outer_step(TABLE, th, b, reps, alpha=1.3, eta=0.7, mu=0.9)
    out = variants.isoloco_outer_step_variant(TABLE, th, b, reps, alpha=1.3, eta=0.7, mu=0.9)
    for key in ("theta", "momentum", "update"):
        assert np.allclose(out[key], ref[key], rtol=1e-12, atol=1e-15)
    assert np.allclose(out["sigma_bar"][:2], ref["sigma_bar"][:2], rtol=1e-12)


@pytest.mark.parametrize("orth,mom_kind", [(0, 1), (1, 0), (1, 1)])
def test_mu_zero_is_eq2_for_every_momentum_choice(orth, mom_kind):
    th, b, reps = _inputs(2)
    base = variants.isoloco_outer_step_variant(TABLE, th, b, reps, alpha=1.0, eta=0.7, mu=0.0)
    out = variants.isoloco_outer_step_variant(TABLE, th, b, reps, alpha=1.0, eta=0.7, mu=0.0,
                                              orth_target=orth, momentum_kind=mom_kind)
    assert np.allclose(out["theta"], base["theta"], rtol=1e-12, atol=1e-15)
    # and Eq. 2: theta' = theta - eta * U
    assert np.allclose(out["theta"], th.astype(np.float64) - 0.7 * base["update"], rtol=1e-12, atol=1e-15)


def _aligned(c, b_scale):
    """A single 8 x 5 matrix: Delta = c Q0 (replica = theta - c Q0), B = b_scale Q0.  The
    replicas are float32, so Delta is c Q0 to ~1e-7 and its polar factor Q0 to ~1e-7."""
    q0, _ = np.linalg.qr(np.random.default_rng(3).standard_normal((8, 5)))
    theta = np.zeros(40, np.float32)
    reps = (theta - (c * q0).ravel()).astype(np.float32)[None]
    mom = (b_scale * q0).ravel().astype(np.float32)
    # the float32 inputs carry the exact data both sides see
    d = (theta.astype(np.float64) - reps[0].astype(np.float64)).reshape(8, 5)
    return [(0, 8, 5)], theta, mom, reps, d, mom.astype(np.float64).reshape(8, 5)


def test_orthogonalised_momentum_update_closed_form():
    table, th, b, reps, d, bm = _aligned(0.3, 0.05)
    mu, eta = 0.9, 0.7
    out = variants.isoloco_outer_step_variant(table, th, b, reps, alpha=1.0, eta=eta, mu=mu, orth_target=1)
    # P = D + mu (mu B + D) is again a multiple of the same Q0, so Iso(P) = P
    p = d + mu * (mu * bm + d)
    assert np.allclose(out["update"].reshape(8, 5), p, rtol=1e-6, atol=0)
    assert np.allclose(out["momentum"].reshape(8, 5), mu * bm + d, rtol=1e-12, atol=1e-15)
    assert np.allclose(out["theta"], -eta * p.ravel(), rtol=1e-6, atol=0)


def test_spectral_scale_closed_form():
    table, th, b, reps, d, bm = _aligned(0.3, 0.0)
    out = variants.isoloco_outer_step_variant(table, th, b, reps, alpha=2.0, eta=0.7, mu=0.0, scale_kind=1)
    q0 = d / 0.3
    assert np.allclose(out["update"].reshape(8, 5), 2.0 * np.sqrt(8 / 5) * q0, rtol=1e-6, atol=0)


def test_standard_momentum_hand_worked_scalar():
    """Delta = 1 twice, B0 = 0, eta = 0.7, mu = 0.9: B1 = 1, theta -= 0.7; B2 = 1.9, theta -= 1.33."""
    table = [(0, 1, 0)]
    b, th = np.zeros(1, np.float32), np.zeros(1, np.float32)
    reps = np.array([[-1.0]], np.float32)                  # theta - replica = 1
    out1 = variants.isoloco_outer_step_variant(table, th, b, reps, eta=0.7, mu=0.9, momentum_kind=1)
    assert out1["momentum"][0] == pytest.approx(1.0) and out1["theta"][0] == pytest.approx(-0.7)
    th2 = out1["theta"].astype(np.float32)
    out2 = variants.isoloco_outer_step_variant(table, th2, out1["momentum"].astype(np.float32), th2[None] - 1.0,
                                               eta=0.7, mu=0.9, momentum_kind=1)
    assert out2["momentum"][0] == pytest.approx(1.9) and out2["theta"][0] == pytest.approx(-0.7 - 1.33)


def test_excluding_a_matrix_is_a_table_choice():
    """A 2-D tensor listed as 1-D gets plain Delta through Nesterov, like DiLoCo's step."""
    th, b, reps = _inputs(4)
    table = [(0, 24, 0), (24, 3, 5), (39, 5, 0)]
    out = variants.isoloco_outer_step_variant(table, th, b, reps, alpha=1.0, eta=0.7, mu=0.9)
    dil = oracle.diloco_outer_step(th, b, reps, eta=0.7, mu=0.9)
    assert np.allclose(out["theta"][:24], dil["theta"][:24], rtol=1e-12, atol=1e-15)


# ---------------------------------------------------------------- clip_high / clip_low (Sec. 4.5)
def test_clip_diagonal_worked_example():
    """Singular values 3, 1, 2 (mean 2): clip_high -> 2, 1, 2; clip_low -> 3, 2, 2."""
    d = np.zeros((4, 3))
    d[0, 0], d[1, 1], d[2, 2] = 3.0, 1.0, 2.0
    hi, sb = variants.clip_spectrum(d, 1)
    lo, _ = variants.clip_spectrum(d, 2)
    assert sb == pytest.approx(2.0, rel=1e-14)
    want_hi = np.zeros((4, 3)); want_hi[0, 0], want_hi[1, 1], want_hi[2, 2] = 2.0, 1.0, 2.0
    want_lo = np.zeros((4, 3)); want_lo[0, 0], want_lo[1, 1], want_lo[2, 2] = 3.0, 2.0, 2.0
    assert np.allclose(hi, want_hi, atol=1e-13) and np.allclose(lo, want_lo, atol=1e-13)


@pytest.mark.parametrize("shape", [(7, 4), (3, 6), (5, 5)])
def test_clip_high_plus_clip_low_is_delta_plus_iso_c(shape):
    """min(s, m) + max(s, m) = s + m for every singular value."""
    d = np.random.default_rng(sum(shape)).standard_normal(shape)
    hi, _ = variants.clip_spectrum(d, 1)
    lo, _ = variants.clip_spectrum(d, 2)
    iso, _ = oracle.iso_c(d, 1.0)
    assert np.allclose(hi + lo, d + iso, rtol=0, atol=1e-12)


@pytest.mark.parametrize("kind", [1, 2])
def test_clip_spectrum_against_lapack(kind):
    d = np.random.default_rng(7 + kind).standard_normal((9, 6)) @ np.diag([5, 3, 1, 0.5, 0.2, 0.1])
    out, sb = variants.clip_spectrum(d, kind)
    s = np.linalg.svd(d, compute_uv=False)
    assert sb == pytest.approx(s.mean(), rel=1e-12)
    want = np.sort(np.minimum(s, sb) if kind == 1 else np.maximum(s, sb))
    assert np.allclose(np.sort(np.linalg.svd(out, compute_uv=False)), want, rtol=1e-12)
    # the singular vectors are Delta's: out^T Delta is symmetric
    h = out.T @ d
    assert np.allclose(h, h.T, atol=1e-12)


@pytest.mark.parametrize("kind", [1, 2])
def test_clip_orthogonal_equivariance_and_fixed_points(kind):
    rng = np.random.default_rng(11)
    d = rng.standard_normal((6, 4))
    p, _ = np.linalg.qr(rng.standard_normal((6, 6)))
    w, _ = np.linalg.qr(rng.standard_normal((4, 4)))
    a, _ = variants.clip_spectrum(p @ d @ w, kind)
    b, _ = variants.clip_spectrum(d, kind)
    assert np.allclose(a, p @ b @ w, atol=1e-12)
    q, _ = np.linalg.qr(rng.standard_normal((6, 4)))
    c, _ = variants.clip_spectrum(0.3 * q, kind)          # equal singular values: unchanged
    assert np.allclose(c, 0.3 * q, atol=1e-13)


@pytest.mark.parametrize("kind", [1, 2])
def test_clip_outer_step_sgd(kind):
    th, b, reps = _inputs(5)
    out = variants.isoloco_outer_step_variant(TABLE, th, b, reps, alpha=1.3, eta=0.7, mu=0.0, spectrum_kind=kind)
    d = oracle.pseudo_gradient(th, reps)
    for i, (off, r, c) in enumerate(TABLE):
        sl = slice(off, off + r * (c or 1))
        want = 1.3 * variants.clip_spectrum(d[sl].reshape(r, c), kind)[0].ravel() if c else d[sl]
        assert np.allclose(out["update"][sl], want, rtol=1e-12, atol=1e-15)
    assert np.allclose(out["theta"], th.astype(np.float64) - 0.7 * out["update"], rtol=1e-12, atol=1e-15)
