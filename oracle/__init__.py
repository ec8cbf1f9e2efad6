"""fp64 CPU oracle for the IsoLoCo / DiLoCo outer step (test infrastructure).

This package is TEST INFRASTRUCTURE.  It restates what the outer step of
"Can Model Merging Improve Aggregation in DiLoCo?" (arXiv 2607.03011) computes,
in plain double precision on the CPU:

* Alg. 1 -- DiLoCo: mean pseudo-gradient, Nesterov SGD as the outer optimiser.
* Alg. 2 -- IsoLoCo: Iso-C (SVD, every singular value replaced by their mean)
  on each 2-D tensor of the mean pseudo-gradient, then Nesterov momentum.
* Sec. 2.2 / Eq. 1 -- Iso-C model merging of task vectors.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg
may import it.  It shares no code with the CUDA library; the C source
(``isoloco_oracle.c``) is compiled here with gcc into ``oracle/_build``.

Parity status: pinned (see ``tests/test_oracle_pins.py``).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "isoloco_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

_c_i64p = ctypes.POINTER(ctypes.c_int64)
_c_ip = ctypes.POINTER(ctypes.c_int)
_c_dp = ctypes.POINTER(ctypes.c_double)
_c_fp = ctypes.POINTER(ctypes.c_float)
_c_vpp = ctypes.POINTER(ctypes.c_void_p)


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, OpenMP, IEEE semantics kept)."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared",
           "-fno-fast-math", "-ffp-contract=off", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            path = build()
            lib = ctypes.CDLL(path)
            lib.orc_num_threads.restype = ctypes.c_int
            lib.orc_svd.argtypes = [ctypes.c_int, ctypes.c_int, _c_dp, _c_dp, _c_dp, _c_dp, _c_ip]
            lib.orc_svd.restype = ctypes.c_int
            lib.orc_iso_c.argtypes = [ctypes.c_int, ctypes.c_int, _c_dp, ctypes.c_double,
                                      _c_dp, _c_dp, _c_ip]
            lib.orc_iso_c.restype = ctypes.c_int
            lib.orc_pseudo_gradient.argtypes = [ctypes.c_int64, _c_fp, _c_vpp, ctypes.c_int,
                                                ctypes.c_int, ctypes.c_int, _c_dp]
            lib.orc_pseudo_gradient.restype = None
            lib.orc_nesterov.argtypes = [ctypes.c_int64, _c_dp, ctypes.c_double,
                                         ctypes.c_double, _c_dp, _c_dp, _c_dp, _c_dp]
            lib.orc_nesterov.restype = None
            lib.orc_isoloco_outer_step.argtypes = [
                _c_i64p, _c_ip, _c_ip, ctypes.c_int, ctypes.c_int64, _c_fp, _c_fp, _c_vpp,
                ctypes.c_int, ctypes.c_int, ctypes.c_double, ctypes.c_double, ctypes.c_double,
                ctypes.c_int, _c_ip, _c_dp, _c_dp, _c_dp, _c_dp, _c_ip]
            lib.orc_isoloco_outer_step.restype = ctypes.c_int
            lib.orc_diloco_outer_step.argtypes = [
                ctypes.c_int64, _c_fp, _c_fp, _c_vpp, ctypes.c_int, ctypes.c_int,
                ctypes.c_double, ctypes.c_double, ctypes.c_int, _c_dp, _c_dp]
            lib.orc_diloco_outer_step.restype = ctypes.c_int
            lib.orc_iso_c_merge.argtypes = [
                _c_i64p, _c_ip, _c_ip, ctypes.c_int, ctypes.c_int64, _c_fp, _c_vpp,
                ctypes.c_int, ctypes.c_int, ctypes.c_double, _c_ip, _c_dp, _c_dp]
            lib.orc_iso_c_merge.restype = ctypes.c_int
            _lib = lib
    return _lib


def _p(a, ctype):
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def num_threads() -> int:
    """OpenMP threads the oracle uses (OMP_NUM_THREADS, else all cores)."""
    return int(_load().orc_num_threads())


class OracleError(RuntimeError):
    pass


def _check(rc: int, what: str):
    if rc != 0:
        raise OracleError(f"{what}: oracle status {rc}")


# ----------------------------------------------------------------------------
# Single-matrix routines
# ----------------------------------------------------------------------------
def svd(a: np.ndarray):
    """Thin SVD by one-sided Jacobi: returns (U [m,r], S [r], V [n,r]), A = U diag(S) V^T.

    Singular values come unsorted (the order the Jacobi rotations leave them).
    """
    a = np.ascontiguousarray(a, dtype=np.float64)
    m, n = a.shape
    r = min(m, n)
    u = np.zeros((m, r)); s = np.zeros(r); v = np.zeros((n, r))
    sweeps = ctypes.c_int(0)
    rc = _load().orc_svd(m, n, _p(a, ctypes.c_double), _p(u, ctypes.c_double),
                         _p(s, ctypes.c_double), _p(v, ctypes.c_double), ctypes.byref(sweeps))
    _check(rc, "svd")
    return u, s, v


def iso_c(delta: np.ndarray, alpha: float = 1.0):
    """Iso-C of one matrix (Alg. 2, dim == 2 branch): returns (alpha*sigma_bar*U V^T, sigma_bar)."""
    d = np.ascontiguousarray(delta, dtype=np.float64)
    m, n = d.shape
    out = np.zeros((m, n))
    sb = ctypes.c_double(0.0)
    sweeps = ctypes.c_int(0)
    rc = _load().orc_iso_c(m, n, _p(d, ctypes.c_double), float(alpha), _p(out, ctypes.c_double),
                           ctypes.byref(sb), ctypes.byref(sweeps))
    _check(rc, "iso_c")
    return out, sb.value


def nesterov(u: np.ndarray, theta: np.ndarray, b: np.ndarray, eta: float, mu: float):
    """Alg. 2's Nesterov update: returns (theta', B')."""
    u = np.ascontiguousarray(u, dtype=np.float64).ravel()
    th = np.ascontiguousarray(theta, dtype=np.float64).ravel()
    bb = np.ascontiguousarray(b, dtype=np.float64).ravel()
    to = np.zeros_like(th); bo = np.zeros_like(bb)
    _load().orc_nesterov(u.size, _p(u, ctypes.c_double), float(mu), float(eta),
                         _p(th, ctypes.c_double), _p(bb, ctypes.c_double),
                         _p(to, ctypes.c_double), _p(bo, ctypes.c_double))
    return to, bo


def _rep_ptrs(replicas):
    """Replicas as numpy arrays (float32, or uint16 holding bf16 bits)."""
    reps = [np.ascontiguousarray(r) for r in replicas]
    dts = {r.dtype for r in reps}
    if len(dts) != 1:
        raise ValueError("replicas must share one dtype")
    dt = dts.pop()
    if dt == np.float32:
        code = 0
    elif dt == np.uint16:
        code = 1
    else:
        raise ValueError("replicas must be float32 or uint16 (bf16 bits)")
    arr = (ctypes.c_void_p * len(reps))(*[r.ctypes.data for r in reps])
    return reps, arr, code


def pseudo_gradient(theta: np.ndarray, replicas, mode: int = 0) -> np.ndarray:
    """mode 0: mean(theta - theta_k); 1: sum(theta - theta_k); 2: sum(theta_k - theta)."""
    th = np.ascontiguousarray(theta, dtype=np.float32).ravel()
    reps, arr, code = _rep_ptrs(replicas)
    out = np.zeros(th.size)
    _load().orc_pseudo_gradient(th.size, _p(th, ctypes.c_float), arr, len(reps), code, mode,
                                _p(out, ctypes.c_double))
    return out


# ----------------------------------------------------------------------------
# Whole outer steps over a parameter table
# ----------------------------------------------------------------------------
def _table(table):
    offs = np.ascontiguousarray([t[0] for t in table], dtype=np.int64)
    rows = np.ascontiguousarray([t[1] for t in table], dtype=np.int32)
    cols = np.ascontiguousarray([t[2] for t in table], dtype=np.int32)
    return offs, rows, cols


def _mask(table, only):
    if only is None:
        return None
    m = np.zeros(len(table), dtype=np.int32)
    m[list(only)] = 1
    return m


def isoloco_outer_step(table, theta, momentum, replicas, alpha=1.0, eta=0.7, mu=0.9,
                       reduce_mean=True, only=None):
    """Alg. 2 over a parameter table [(offset, rows, cols)], cols == 0 for 1-D.

    Returns dict(theta, momentum, update, sigma_bar, sweeps); entries of
    parameters outside ``only`` (an index list) are left as NaN.
    """
    offs, rows, cols = _table(table)
    th = np.ascontiguousarray(theta, dtype=np.float32).ravel()
    bb = np.ascontiguousarray(momentum, dtype=np.float32).ravel()
    reps, arr, code = _rep_ptrs(replicas)
    n = th.size
    to = np.full(n, np.nan); bo = np.full(n, np.nan); uo = np.full(n, np.nan)
    sb = np.zeros(len(table)); sw = np.zeros(len(table), dtype=np.int32)
    mask = _mask(table, only)
    rc = _load().orc_isoloco_outer_step(
        _p(offs, ctypes.c_int64), _p(rows, ctypes.c_int), _p(cols, ctypes.c_int), len(table),
        n, _p(th, ctypes.c_float), _p(bb, ctypes.c_float), arr, len(reps), code,
        float(alpha), float(eta), float(mu), int(bool(reduce_mean)),
        None if mask is None else _p(mask, ctypes.c_int),
        _p(to, ctypes.c_double), _p(bo, ctypes.c_double), _p(uo, ctypes.c_double),
        _p(sb, ctypes.c_double), _p(sw, ctypes.c_int))
    _check(rc, "isoloco_outer_step")
    return {"theta": to, "momentum": bo, "update": uo, "sigma_bar": sb, "sweeps": sw}


def diloco_outer_step(theta, momentum, replicas, eta=0.7, mu=0.9, reduce_mean=True):
    """Alg. 1 with Nesterov SGD as OuterOpt.  Returns dict(theta, momentum)."""
    th = np.ascontiguousarray(theta, dtype=np.float32).ravel()
    bb = np.ascontiguousarray(momentum, dtype=np.float32).ravel()
    reps, arr, code = _rep_ptrs(replicas)
    to = np.zeros(th.size); bo = np.zeros(th.size)
    rc = _load().orc_diloco_outer_step(th.size, _p(th, ctypes.c_float), _p(bb, ctypes.c_float),
                                       arr, len(reps), code, float(eta), float(mu),
                                       int(bool(reduce_mean)), _p(to, ctypes.c_double),
                                       _p(bo, ctypes.c_double))
    _check(rc, "diloco_outer_step")
    return {"theta": to, "momentum": bo}


def iso_c_merge(table, base, experts, alpha=1.0, only=None):
    """Iso-C merge of K experts into base.  Returns dict(out, sigma_bar)."""
    offs, rows, cols = _table(table)
    b = np.ascontiguousarray(base, dtype=np.float32).ravel()
    reps, arr, code = _rep_ptrs(experts)
    out = np.full(b.size, np.nan)
    sb = np.zeros(len(table))
    mask = _mask(table, only)
    rc = _load().orc_iso_c_merge(
        _p(offs, ctypes.c_int64), _p(rows, ctypes.c_int), _p(cols, ctypes.c_int), len(table),
        b.size, _p(b, ctypes.c_float), arr, len(reps), code, float(alpha),
        None if mask is None else _p(mask, ctypes.c_int), _p(out, ctypes.c_double),
        _p(sb, ctypes.c_double))
    _check(rc, "iso_c_merge")
    return {"out": out, "sigma_bar": sb}
