"""Pins for the fp64 oracle: values fixed by the paper's definitions and by mathematics.

Each check is independent of the oracle's own code: closed forms, invariants,
special cases, an independent scaled-Newton polar iteration, a library SVD, and
hand-worked examples under tests/golden/.  Together they are meant to catch a
dropped term, a wrong sign or index, or a transposed operand anywhere in the
oracle (Jacobi SVD, Householder QR, Iso-C, the pseudo-gradient reduction and the
Nesterov update).
"""
import numpy as np
import pytest

import oracle
from conftest import read_golden

RNG = np.random.default_rng(1234)


def lowrank_plus_noise(m, n, r=4, shared=1.0, noise=0.5, rng=RNG):
    a = rng.standard_normal((m, r))
    b = rng.standard_normal((n, r))
    return a @ b.T * (shared / np.sqrt(r)) + noise * rng.standard_normal((m, n))


def np_iso_c(d, alpha=1.0):
    u, s, vt = np.linalg.svd(d, full_matrices=False)
    return alpha * s.mean() * (u @ vt), s.mean()


def higham_polar(a, iters=100):
    """Independent polar factor: Higham's scaled Newton iteration (square, nonsingular)."""
    x = a.copy()
    for _ in range(iters):
        xi = np.linalg.inv(x)
        zeta = np.sqrt(np.linalg.norm(xi) / np.linalg.norm(x))
        xn = 0.5 * (zeta * x + xi.T / zeta)
        if np.linalg.norm(xn - x) <= 1e-15 * np.linalg.norm(xn):
            return xn
        x = xn
    return x


# --------------------------------------------------------------------------
# Closed forms and hand-worked examples
# --------------------------------------------------------------------------
def test_iso_c_2x2_golden():
    for (a, sb, iso) in read_golden("iso_c_2x2.txt"):
        A = np.array(a).reshape(2, 2)
        out, sigma_bar = oracle.iso_c(A)
        assert sigma_bar == pytest.approx(sb[0], rel=1e-14)
        np.testing.assert_allclose(out, np.array(iso).reshape(2, 2), rtol=0, atol=1e-13)


@pytest.mark.parametrize("seed", range(8))
def test_iso_c_2x2_closed_form(seed):
    rng = np.random.default_rng(seed)
    A = rng.standard_normal((2, 2)) * 10 ** rng.uniform(-6, 3)
    det = A[0, 0] * A[1, 1] - A[0, 1] * A[1, 0]
    cof = np.array([[A[1, 1], -A[1, 0]], [-A[0, 1], A[0, 0]]])
    tsum = np.sqrt((A ** 2).sum() + 2 * abs(det))          # sigma_1 + sigma_2
    Q = (A + np.sign(det) * cof) / tsum
    alpha = 1.7
    out, sb = oracle.iso_c(A, alpha)
    assert sb == pytest.approx(tsum / 2, rel=1e-13)
    np.testing.assert_allclose(out, alpha * (tsum / 2) * Q, rtol=0, atol=1e-12 * abs(alpha * tsum))
    u, s, v = oracle.svd(A)
    assert s.sum() == pytest.approx(tsum, rel=1e-13)


def test_nesterov_scalar_golden():
    rows = read_golden("nesterov_scalar.txt")
    theta, b = np.zeros(1), np.zeros(1)
    for (vals,) in rows:
        step, b_exp, p_exp, th_exp = vals
        theta_new, b = oracle.nesterov(np.ones(1), theta, b, eta=0.7, mu=0.9)
        p = (theta - theta_new) / 0.7
        theta = theta_new
        assert b[0] == pytest.approx(b_exp, abs=1e-14)
        assert p[0] == pytest.approx(p_exp, abs=1e-14)
        assert theta[0] == pytest.approx(th_exp, abs=1e-14)


# --------------------------------------------------------------------------
# SVD and Iso-C invariants
# --------------------------------------------------------------------------
SHAPES = [(1, 1), (1, 9), (9, 1), (3, 2), (2, 3), (17, 17), (64, 64), (65, 130), (130, 65),
          (256, 64), (64, 256), (300, 7)]


@pytest.mark.parametrize("m,n", SHAPES)
def test_svd_reconstructs_and_matches_library(m, n):
    A = lowrank_plus_noise(m, n)
    U, S, V = oracle.svd(A)
    r = min(m, n)
    np.testing.assert_allclose(U @ np.diag(S) @ V.T, A, atol=1e-12 * np.abs(A).max())
    np.testing.assert_allclose(U.T @ U, np.eye(r), atol=1e-12)
    np.testing.assert_allclose(V.T @ V, np.eye(r), atol=1e-12)
    np.testing.assert_allclose(np.sort(S)[::-1], np.linalg.svd(A, compute_uv=False),
                               rtol=1e-11, atol=1e-13 * S.max())


@pytest.mark.parametrize("m,n", SHAPES)
def test_iso_c_spectrum_is_flat(m, n):
    """Every singular value of the output equals alpha * sigma_bar (Alg. 2)."""
    D = lowrank_plus_noise(m, n)
    alpha = 0.8
    out, sb = oracle.iso_c(D, alpha)
    r = min(m, n)
    G = out.T @ out if m >= n else out @ out.T
    np.testing.assert_allclose(G, (alpha * sb) ** 2 * np.eye(r), atol=1e-12 * (alpha * sb) ** 2)
    # sigma_bar = ||D||_* / r, and the nuclear norm is carried over exactly
    nuc = np.linalg.svd(D, compute_uv=False).sum()
    assert sb == pytest.approx(nuc / r, rel=1e-12)
    assert np.linalg.svd(out, compute_uv=False).sum() == pytest.approx(alpha * nuc, rel=1e-12)


@pytest.mark.parametrize("m,n", SHAPES)
def test_iso_c_matches_library_svd(m, n):
    D = lowrank_plus_noise(m, n)
    out, sb = oracle.iso_c(D, 1.3)
    ref, sb_ref = np_iso_c(D, 1.3)
    assert sb == pytest.approx(sb_ref, rel=1e-12)
    np.testing.assert_allclose(out, ref, atol=1e-11 * np.abs(ref).max())


@pytest.mark.parametrize("n", [2, 5, 32, 96])
def test_polar_matches_scaled_newton(n):
    A = lowrank_plus_noise(n, n, r=2, noise=0.3)
    out, sb = oracle.iso_c(A, 1.0)
    Q = higham_polar(A)
    np.testing.assert_allclose(out / sb, Q, atol=1e-11)
    # singular values from an independent symmetric eigen-solve of A^T A
    ev = np.sqrt(np.clip(np.linalg.eigvalsh(A.T @ A), 0, None))
    assert sb == pytest.approx(ev.mean(), rel=1e-9)


@pytest.mark.parametrize("m,n", [(40, 40), (90, 30), (30, 90)])
def test_h_symmetric_psd_trace_is_nuclear_norm(m, n):
    D = lowrank_plus_noise(m, n)
    out, sb = oracle.iso_c(D, 1.0)
    Q = out / sb
    H = Q.T @ D if m >= n else D @ Q.T
    np.testing.assert_allclose(H, H.T, atol=1e-12 * np.abs(H).max())
    assert np.linalg.eigvalsh((H + H.T) / 2).min() > -1e-10 * np.abs(H).max()
    nuc = np.linalg.svd(D, compute_uv=False).sum()
    assert np.trace(H) == pytest.approx(nuc, rel=1e-12)
    assert sb == pytest.approx(np.trace(H) / min(m, n), rel=1e-12)


def test_c_times_orthogonal_is_fixed():
    Q0, _ = np.linalg.qr(RNG.standard_normal((50, 20)))
    for c in (3e-5, 1.0, 7.5):
        out, sb = oracle.iso_c(c * Q0, 2.0)
        assert sb == pytest.approx(c, rel=1e-13)
        np.testing.assert_allclose(out, 2.0 * c * Q0, atol=1e-13 * c)
        # RMS of the spectrum equals its mean only here (Sec. 4.3 remark)
        s = oracle.svd(c * Q0)[1]
        assert np.sqrt((s ** 2).mean()) == pytest.approx(s.mean(), rel=1e-13)


def test_diagonal_and_vectors():
    d = np.array([3.0, -0.5, 2.0, -7.0])
    out, sb = oracle.iso_c(np.diag(d), 1.0)
    assert sb == pytest.approx(np.abs(d).mean(), rel=1e-14)
    np.testing.assert_allclose(out, np.abs(d).mean() * np.diag(np.sign(d)), atol=1e-14)
    row = RNG.standard_normal((1, 37))
    out, sb = oracle.iso_c(row, 0.6)
    np.testing.assert_allclose(out, 0.6 * row, atol=1e-14)
    assert sb == pytest.approx(np.linalg.norm(row), rel=1e-14)
    col = RNG.standard_normal((23, 1))
    out, _ = oracle.iso_c(col, 1.0)
    np.testing.assert_allclose(out, col, atol=1e-14)


def test_rms_exceeds_mean_on_generic_spectra():
    D = lowrank_plus_noise(64, 48)
    s = oracle.svd(D)[1]
    assert np.sqrt((s ** 2).mean()) > s.mean() * (1 + 1e-6)


def test_homogeneity_transpose_equivariance():
    D = lowrank_plus_noise(33, 21)
    base, _ = oracle.iso_c(D)
    np.testing.assert_allclose(oracle.iso_c(4.0 * D)[0], 4.0 * base, atol=1e-12)
    np.testing.assert_allclose(oracle.iso_c(-D)[0], -base, atol=1e-13)
    np.testing.assert_allclose(oracle.iso_c(D.T)[0], base.T, atol=1e-13)
    P, _ = np.linalg.qr(RNG.standard_normal((33, 33)))
    R, _ = np.linalg.qr(RNG.standard_normal((21, 21)))
    np.testing.assert_allclose(oracle.iso_c(P @ D @ R)[0], P @ base @ R, atol=1e-12)


def test_rank_deficient_is_partial_isometry():
    m, n, rho = 30, 20, 6
    D = RNG.standard_normal((m, rho)) @ RNG.standard_normal((rho, n))
    out, sb = oracle.iso_c(D, 1.0)
    s_out = np.linalg.svd(out, compute_uv=False)
    assert np.sum(s_out > 1e-8 * s_out.max()) == rho
    nuc = np.linalg.svd(D, compute_uv=False).sum()
    assert s_out.sum() == pytest.approx(nuc * rho / n, rel=1e-10)


def _np_partial_isometry(d, alpha=1.0):
    """Iso-C of a rank-deficient matrix from LAPACK's SVD: alpha * mean(sigma) * U_rho V_rho^T
    with rho the singular values above r * eps * sigma_max (reading C3)."""
    u, s, vt = np.linalg.svd(d, full_matrices=False)
    rho = int(np.sum(s > min(d.shape) * np.finfo(float).eps * s[0]))
    return alpha * s.mean() * (u[:, :rho] @ vt[:rho]), s.mean(), rho


@pytest.mark.parametrize("m,n,zero", [(128, 64, ("rows", 5)), (64, 128, ("cols", 7)), (96, 40, ("cols", 25)),
                                      (256, 256, ("rows", 240)), (200, 200, ("both", 150))])
def test_structurally_rank_deficient(m, n, zero):
    """Zero rows or columns (entries no worker touched) give an exactly rank-deficient
    matrix; rounding-level columns must not keep the Jacobi sweeps going, and the result
    is LAPACK's partial isometry with rho = the number of nonzero rows (columns)."""
    rng = np.random.default_rng(m * 1000 + n)
    D = rng.standard_normal((m, n))
    kind, keep = zero
    if kind in ("rows", "both"):
        D[keep:, :] = 0.0
    if kind in ("cols", "both"):
        D[:, keep:] = 0.0
    out, sb = oracle.iso_c(D, 0.5)
    ref, sb_ref, rho = _np_partial_isometry(D, 0.5)
    assert rho == keep
    assert sb == pytest.approx(sb_ref, rel=1e-12)
    assert np.linalg.norm(out - ref) / np.linalg.norm(ref) < 1e-11
    s_out = np.linalg.svd(out, compute_uv=False)
    assert np.all(np.abs(s_out[:rho] / (0.5 * sb) - 1.0) < 1e-11) and np.all(s_out[rho:] < 1e-12 * s_out[0])


def test_low_rank_product_is_partial_isometry():
    """A generic rank-12 product (no zero rows) of a 300 x 200 matrix."""
    rng = np.random.default_rng(7)
    D = rng.standard_normal((300, 12)) @ rng.standard_normal((12, 200))
    out, sb = oracle.iso_c(D)
    ref, sb_ref, rho = _np_partial_isometry(D)
    assert rho == 12
    assert sb == pytest.approx(sb_ref, rel=1e-10)
    assert np.linalg.norm(out - ref) / np.linalg.norm(ref) < 1e-9


def test_zero_matrix():
    out, sb = oracle.iso_c(np.zeros((8, 5)), 1.0)
    assert sb == 0.0 and not out.any()


def test_ill_conditioned_generator_like():
    """kappa ~ 1e5 low-rank-plus-small-noise matrix: still exact to ~1e-10."""
    D = lowrank_plus_noise(256, 256, r=8, shared=1.0, noise=1e-3)
    out, sb = oracle.iso_c(D)
    ref, sb_ref = np_iso_c(D)
    assert sb == pytest.approx(sb_ref, rel=1e-11)
    assert np.linalg.norm(out - ref) / np.linalg.norm(ref) < 1e-9


# --------------------------------------------------------------------------
# Reduction, whole steps, and the paper's identities
# --------------------------------------------------------------------------
def _tiny_inputs(K=3, dtype=np.float32, seed=5):
    rng = np.random.default_rng(seed)
    table = [(0, 12, 8), (96, 8, 12), (192, 10, 0), (202, 5, 5), (227, 1, 0)]
    N = 228
    theta = (0.02 * rng.standard_normal(N)).astype(np.float32)
    mom = (1e-4 * rng.standard_normal(N)).astype(np.float32)
    reps = [(theta - 1e-3 * rng.standard_normal(N)).astype(np.float32) for _ in range(K)]
    return table, theta, mom, reps


def test_pseudo_gradient_modes():
    table, theta, mom, reps = _tiny_inputs()
    d64 = [theta.astype(np.float64) - r.astype(np.float64) for r in reps]
    np.testing.assert_allclose(oracle.pseudo_gradient(theta, reps, 0), np.mean(d64, axis=0),
                               rtol=1e-15, atol=0)
    np.testing.assert_allclose(oracle.pseudo_gradient(theta, reps, 1), np.sum(d64, axis=0),
                               rtol=1e-15, atol=0)
    np.testing.assert_allclose(oracle.pseudo_gradient(theta, reps, 2), -np.sum(d64, axis=0),
                               rtol=1e-15, atol=0)


def test_bf16_replicas_upcast_exactly():
    table, theta, mom, reps = _tiny_inputs()
    bits = [(r.view(np.uint32) >> 16).astype(np.uint16) for r in reps]   # truncate to bf16
    vals = [(b.astype(np.uint32) << 16).view(np.float32).astype(np.float64) for b in bits]
    ref = np.mean([theta.astype(np.float64) - v for v in vals], axis=0)
    np.testing.assert_array_equal(oracle.pseudo_gradient(theta, bits, 0), ref)


def _np_isoloco(table, theta, mom, reps, alpha, eta, mu):
    """Alg. 2 written with numpy's SVD, as an independent check of the whole step."""
    D = np.mean([theta.astype(np.float64) - r.astype(np.float64) for r in reps], axis=0)
    U = D.copy()
    for (o, r, c) in table:
        if c > 0:
            U[o:o + r * c] = np_iso_c(D[o:o + r * c].reshape(r, c), alpha)[0].ravel()
    b = mu * mom.astype(np.float64) + U
    th = theta.astype(np.float64) - eta * (U + mu * b)
    return th, b, U


def test_isoloco_step_matches_numpy_restatement():
    table, theta, mom, reps = _tiny_inputs()
    res = oracle.isoloco_outer_step(table, theta, mom, reps, alpha=1.4, eta=1.8, mu=0.8)
    th, b, U = _np_isoloco(table, theta, mom, reps, 1.4, 1.8, 0.8)
    np.testing.assert_allclose(res["update"], U, atol=1e-15)
    np.testing.assert_allclose(res["momentum"], b, atol=1e-15)
    np.testing.assert_allclose(res["theta"], th, atol=1e-15)


def test_one_dim_params_ignore_alpha_and_take_the_mean():
    table, theta, mom, reps = _tiny_inputs()
    a = oracle.isoloco_outer_step(table, theta, mom, reps, alpha=1.0)
    b = oracle.isoloco_outer_step(table, theta, mom, reps, alpha=3.0)
    D = oracle.pseudo_gradient(theta, reps, 0)
    for (o, r, c) in table:
        sl = slice(o, o + r * (c or 1))
        if c == 0:
            np.testing.assert_array_equal(a["update"][sl], D[sl])
            np.testing.assert_array_equal(a["update"][sl], b["update"][sl])
        else:
            np.testing.assert_allclose(b["update"][sl], 3.0 * a["update"][sl], rtol=1e-12)


def test_sgd_outer_step_is_task_arithmetic():
    """Eq. 2: with mu = 0 the DiLoCo step is theta + (eta/R) sum_i (theta_i - theta)."""
    table, theta, mom, reps = _tiny_inputs(K=4)
    eta = 1.6
    res = oracle.diloco_outer_step(theta, mom, reps, eta=eta, mu=0.0)
    tau = [r.astype(np.float64) - theta.astype(np.float64) for r in reps]
    np.testing.assert_allclose(res["theta"], theta + eta / 4 * np.sum(tau, axis=0), atol=1e-16)
    # and IsoLoCo reduces to DiLoCo on a table with no matrices
    flat = [(0, theta.size, 0)]
    iso = oracle.isoloco_outer_step(flat, theta, mom, reps, eta=eta, mu=0.9)
    dil = oracle.diloco_outer_step(theta, mom, reps, eta=eta, mu=0.9)
    np.testing.assert_array_equal(iso["theta"], dil["theta"])
    np.testing.assert_array_equal(iso["momentum"], dil["momentum"])


def test_iso_c_merge_definition():
    table, theta, mom, reps = _tiny_inputs()
    res = oracle.iso_c_merge(table, theta, reps, alpha=0.5)
    T = np.sum([r.astype(np.float64) - theta.astype(np.float64) for r in reps], axis=0)
    for (o, r, c) in table:
        sl = slice(o, o + r * (c or 1))
        if c == 0:     # Eq. 1: base + lambda * sum tau
            np.testing.assert_allclose(res["out"][sl], theta[sl] + 0.5 * T[sl], atol=1e-16)
        else:
            iso, _ = np_iso_c(T[sl].reshape(r, c), 0.5)
            np.testing.assert_allclose(res["out"][sl], theta[sl] + iso.ravel(), atol=1e-15)


def test_merge_and_step_agree_on_sign_convention():
    """IsoC is odd: the merge of tau = theta_k - theta equals -IsoC(sum Delta)."""
    table, theta, mom, reps = _tiny_inputs()
    m = oracle.iso_c_merge(table, theta, reps, alpha=1.0)
    s = oracle.isoloco_outer_step(table, theta, mom, reps, alpha=1.0, reduce_mean=False)
    np.testing.assert_allclose(m["out"] - theta.astype(np.float64), -s["update"], atol=1e-15)


def test_second_step_reuses_momentum():
    """Checkpoint/resume of the outer state: running step 2 from the saved (theta, B)."""
    table, theta, mom, reps = _tiny_inputs()
    s1 = oracle.isoloco_outer_step(table, theta, np.zeros_like(mom), reps)
    th1 = s1["theta"].astype(np.float32)
    b1 = s1["momentum"].astype(np.float32)
    rng = np.random.default_rng(9)
    reps2 = [(th1 - 1e-3 * rng.standard_normal(th1.size)).astype(np.float32) for _ in reps]
    s2 = oracle.isoloco_outer_step(table, th1, b1, reps2)
    th, b, U = _np_isoloco(table, th1, b1, reps2, 1.0, 0.7, 0.9)
    np.testing.assert_allclose(s2["theta"], th, atol=1e-15)
    np.testing.assert_allclose(s2["momentum"], b, atol=1e-15)


def test_only_mask_skips_params():
    table, theta, mom, reps = _tiny_inputs()
    res = oracle.isoloco_outer_step(table, theta, mom, reps, only=[1])
    o, r, c = table[1]
    assert np.isfinite(res["theta"][o:o + r * c]).all()
    assert np.isnan(res["theta"][:o]).all()
