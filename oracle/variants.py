"""fp64 oracle for the outer-step ablations of Sec. 4.5 and App. B (test infrastructure).

Alg. 2's outer step, with the choices the paper's ablations vary:

* orth_target 0: Iso-C of the pseudo-gradient Delta, then momentum (Alg. 2).
  orth_target 1: momentum first on the raw Delta, B' = mu B + Delta, the update
  P = Delta + mu B' (Nesterov) or P = B' (standard), and Iso-C of P for 2-D tensors;
  theta' = theta - eta * Iso(P) (2-D) or theta - eta * P (1-D).
* momentum_kind 0: Nesterov, B' = mu B + U, theta' = theta - eta (U + mu B') (Alg. 2);
  momentum_kind 1: standard momentum, theta' = theta - eta B'.
* scale_kind 0: the Iso-C scale sigma_bar (mean singular value, or with fast_steps its
  RMS ||X||_F / sqrt(r)); scale_kind 1: Muon's spectral scale sqrt(rows / cols) (App. B).
* fast_steps k > 0: the polar factor by k fixed quintic steps (oracle/fast_ns.py) instead
  of the SVD.
* spectrum_kind 1 (clip_high) / 2 (clip_low), Sec. 4.5: only the singular values above /
  below their mean sigma_bar are set to it, the others kept: U = alpha * U_D diag(f(s)) V_D^T
  with f(s) = min(s, sigma_bar) / max(s, sigma_bar), from the oracle's SVD.  Singular values
  that the SVD finds zero (below r * eps * s_max) stay zero, as in Iso-C's partial isometry.
* Excluding a 2-D tensor from Iso-C (Sec. 4.5) is a table choice: it is listed as a 1-D
  tensor of rows * cols elements and updated with Delta.

Only ``tests/`` may import this module.  It shares no code with the CUDA library; the
reduction and the SVD-based Iso-C are the pinned C oracle's (oracle/isoloco_oracle.c).

Parity status: pinned (``tests/test_oracle_variants.py``: default flags reproduce the
oracle's Alg. 2, mu = 0 collapses every momentum choice to Eq. 2, closed forms on
c * orthogonal inputs, a hand-worked standard-momentum scalar; the clip variants by a
diagonal worked example, clip_high + clip_low = Delta + Iso-C(Delta), their spectra against
LAPACK's, and orthogonal equivariance).
"""
from __future__ import annotations

import numpy as np

from . import fast_ns, iso_c, pseudo_gradient, svd


def _polar_and_sigma(x: np.ndarray, fast_steps: int):
    """(Q, sigma_bar) of one matrix: SVD-based polar factor and mean singular value, or the
    fast variant's fixed-step factor and RMS singular value."""
    if fast_steps:
        q, _ = fast_ns.fast_polar(x, fast_ns.fast_schedule(fast_steps))
        return q, float(np.linalg.norm(x) / np.sqrt(min(x.shape)))
    u, sigma = iso_c(x, 1.0)            # sigma * U V^T and sigma
    q = u / sigma if sigma > 0 else np.zeros_like(u)
    return q, float(sigma)


def clip_spectrum(x: np.ndarray, kind: int):
    """(U diag(f(s)) V^T, sigma_bar) of one matrix, f(s) = min(s, sigma_bar) (kind 1,
    clip_high) or max(s, sigma_bar) (kind 2, clip_low), sigma_bar = sum(s) / min(m, n)."""
    u, s, v = svd(np.asarray(x, dtype=np.float64))
    r = min(x.shape)
    sbar = float(s.sum() / r)
    smax = float(s.max()) if s.size else 0.0
    if not smax > 0.0:
        return np.zeros(x.shape), 0.0
    nz = s > r * np.finfo(np.float64).eps * smax
    f = np.where(nz, np.minimum(s, sbar) if kind == 1 else np.maximum(s, sbar), 0.0)
    return (u * f) @ v.T, sbar


def isoloco_outer_step_variant(table, theta, momentum, replicas, alpha=1.0, eta=0.7, mu=0.9,
                               orth_target=0, momentum_kind=0, scale_kind=0, fast_steps=0,
                               reduce_mean=True, only=None, spectrum_kind=0):
    """Returns dict(theta, momentum, update, sigma_bar) in fp64 (sigma_bar per table entry,
    0 for 1-D tensors); entries of parameters outside ``only`` are NaN."""
    th = np.asarray(theta, dtype=np.float64).ravel()
    bb = np.asarray(momentum, dtype=np.float64).ravel()
    dd = pseudo_gradient(np.asarray(theta, dtype=np.float32), replicas, mode=0 if reduce_mean else 1)
    n = th.size
    to, bo, uo = np.full(n, np.nan), np.full(n, np.nan), np.full(n, np.nan)
    sig = np.zeros(len(table))
    for i, (off, rows, cols) in enumerate(table):
        sl = slice(off, off + rows * (cols if cols > 0 else 1))
        if only is not None and i not in only:
            if cols > 0:
                sig[i] = np.nan
            continue
        d, b = dd[sl], bb[sl]
        if orth_target:
            nb = mu * b + d
            p = d + mu * nb if momentum_kind == 0 else nb
            if cols > 0 and spectrum_kind:
                um, sig[i] = clip_spectrum(p.reshape(rows, cols), spectrum_kind)
                u = alpha * um.ravel()
            elif cols > 0:
                q, sigma = _polar_and_sigma(p.reshape(rows, cols), fast_steps)
                sig[i] = sigma
                u = alpha * (sigma if scale_kind == 0 else np.sqrt(rows / cols)) * q.ravel()
            else:
                u = p
            to[sl] = th[sl] - eta * u
        else:
            if cols > 0 and spectrum_kind:
                um, sig[i] = clip_spectrum(d.reshape(rows, cols), spectrum_kind)
                u = alpha * um.ravel()
            elif cols > 0:
                q, sigma = _polar_and_sigma(d.reshape(rows, cols), fast_steps)
                sig[i] = sigma
                u = alpha * (sigma if scale_kind == 0 else np.sqrt(rows / cols)) * q.ravel()
            else:
                u = d
            nb = mu * b + u
            to[sl] = th[sl] - eta * (u + mu * nb if momentum_kind == 0 else nb)
        bo[sl] = nb
        uo[sl] = u
    return {"theta": to, "momentum": bo, "update": uo, "sigma_bar": sig}
