"""fp64 oracle for the fast IsoLoCo variant of Sec. 4.3 (test infrastructure).

Sec. 4.3 replaces the SVD of Alg. 2 by a fixed, small number of Newton-Schulz-type
steps and the mean singular value by its RMS proxy, sigma_bar ~ ||Delta||_F / sqrt(r).
The paper's own polynomial coefficients are not given in its text; the library's
schedule is ours, so this module restates that schedule from its definition:

* every step applies an odd quintic p(x) = a x + b x^3 + c x^5 to each singular value,
  as X <- X (a I + b X^T X + c (X^T X)^2);
* step t's quintic minimises max |1 - p(x)| over the interval [lo_t, hi_t] that holds
  every singular value at that step, subject to p(x) >= KAPPA x there; solved here as a
  linear program on a grid (scipy's HiGHS);
* the first interval is [1e-3, 1.02] (the iterate is scaled by s = ||Delta^T Delta||_F^{1/2},
  an upper bound of sigma_max); the next interval is the image [min p, max p] widened by a
  relative guard of 2e-3 on each side.

Only ``tests/`` may import this module.  It shares no code with the CUDA library.

Parity status: pinned (``tests/test_oracle_fast.py``: spectral mapping against LAPACK's
SVD, the c * orthogonal closed form, the LP's constraints).
"""
from __future__ import annotations

import numpy as np

ELL = 1e-3
HI = 1.02
GUARD = 2e-3
KAPPA = 0.2
CHAIN = 7   # steps of the chain; a fixed-step run longer than that repeats the last one


def minimax_step(lo: float, hi: float, kappa: float = KAPPA, npts: int = 6000):
    """The odd quintic minimising max |1 - p| on [lo, hi] with p(x) >= kappa x.

    Returns ((a, b, c), error, (min p, max p)) over the grid.
    """
    from scipy.optimize import linprog

    x = np.unique(np.concatenate([np.geomspace(lo, hi, npts), np.linspace(lo, hi, npts)]))
    basis = np.column_stack([x, x ** 3, x ** 5])
    # variables (a, b, c, err): minimise err with -err <= 1 - p(x) <= err, p(x) >= kappa x
    one = np.ones((x.size, 1))
    zero = np.zeros((x.size, 1))
    A = np.vstack([np.hstack([basis, -one]),        # p - 1 <= err
                   np.hstack([-basis, -one]),       # 1 - p <= err
                   np.hstack([-basis, zero])])      # -p <= -kappa x
    b = np.concatenate([np.ones(x.size), -np.ones(x.size), -kappa * x])
    res = linprog(c=[0.0, 0.0, 0.0, 1.0], A_ub=A, b_ub=b,
                  bounds=[(None, None)] * 3 + [(0.0, None)], method="highs")
    if not res.success:
        raise RuntimeError(f"minimax LP failed: {res.message}")
    coef = tuple(float(v) for v in res.x[:3])
    p = basis @ np.asarray(coef)
    return coef, float(res.x[3]), (float(p.min()), float(p.max()))


def schedule(steps: int, ell: float = ELL, hi: float = HI, guard: float = GUARD, kappa: float = KAPPA):
    """The first `steps` quintics of the chain of intervals starting at [ell, hi]."""
    out, lo = [], ell
    for _ in range(steps):
        coef, _, (pmin, pmax) = minimax_step(lo, hi, kappa)
        out.append(coef)
        lo, hi = pmin * (1.0 - guard), pmax * (1.0 + guard)
    return out


def fast_schedule(steps: int):
    """The quintics of a fixed-step run: the chain's first steps, the last one repeated."""
    chain = schedule(min(steps, CHAIN))
    return chain + [chain[-1]] * max(0, steps - CHAIN)


def compose(coefs, x):
    """The composed scalar map f = p_k o ... o p_1 on singular values."""
    y = np.asarray(x, dtype=np.float64)
    for a, b, c in coefs:
        y = a * y + b * y ** 3 + c * y ** 5
    return y


def fast_polar(delta: np.ndarray, coefs):
    """X_k from X_0 = Delta / s by the fixed quintic steps (no convergence test)."""
    d = np.asarray(delta, dtype=np.float64)
    g0 = d.T @ d
    s = np.sqrt(np.sqrt(np.sum(g0 * g0)))
    if not s > 0.0:
        return np.zeros_like(d), 0.0
    x = d / s
    for a, b, c in coefs:
        g = x.T @ x
        x = x @ (a * np.eye(g.shape[0]) + b * g + c * (g @ g))
    return x, s


def fast_iso(delta: np.ndarray, coefs, alpha: float = 1.0):
    """alpha * sigma_rms * X_k and sigma_rms = ||Delta||_F / sqrt(min(m, n))."""
    d = np.asarray(delta, dtype=np.float64)
    r = min(d.shape)
    sigma = float(np.linalg.norm(d) / np.sqrt(r))
    x, _ = fast_polar(d, coefs)
    return alpha * sigma * x, sigma


def isoloco_outer_step_fast(table, theta, momentum, delta, alpha, eta, mu, coefs, only=None):
    """Alg. 2 with Sec. 4.3's fast Iso-C on every 2-D tensor, from a given pseudo-gradient
    (the reduction is the same as the exact path's).  Returns dict(theta, momentum, update,
    sigma_bar) in fp64, sigma_bar per table entry (0 for 1-D); entries outside ``only`` are NaN."""
    th = np.asarray(theta, dtype=np.float64).ravel()
    bb = np.asarray(momentum, dtype=np.float64).ravel()
    dd = np.asarray(delta, dtype=np.float64).ravel()
    n = th.size
    to, bo, uo = np.full(n, np.nan), np.full(n, np.nan), np.full(n, np.nan)
    sig = np.zeros(len(table))
    for i, (off, rows, cols) in enumerate(table):
        ln = rows * (cols if cols > 0 else 1)
        sl = slice(off, off + ln)
        if cols > 0:
            if only is not None and i not in only:
                sig[i] = np.nan
                continue
            u, sbar = fast_iso(dd[sl].reshape(rows, cols), coefs, alpha)
            u = u.ravel()
            sig[i] = sbar
        else:
            if only is not None and i not in only:
                continue
            u = dd[sl]
        nb = mu * bb[sl] + u
        to[sl] = th[sl] - eta * (u + mu * nb)
        bo[sl] = nb
        uo[sl] = u
    return {"theta": to, "momentum": bo, "update": uo, "sigma_bar": sig}
