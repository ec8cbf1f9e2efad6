"""Thin Python binding over the C ABI of libisoloco (include/isoloco.h).

Argument marshalling only: every step of the outer step runs in the CUDA library.
Tensors are torch CUDA tensors (fp32 theta / momentum, fp32 or bf16 replicas); the
binding passes their data pointers and the current CUDA stream across the ABI.
If the library cannot be built or loaded the import of this module fails: there is
no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Optional, Sequence

import torch

from . import _build

PHASES = ["reduce", "gram", "finalize", "control", "poly", "update", "trace", "apply", "diloco", "other", "trim", "clip"]

OK = 0
ERR_INVALID = -1
ERR_ALIGN = -2
ERR_NONFINITE = -3
ERR_NOT_CONVERGED = -4
ERR_CUDA = -5
ERR_OOM = -6
ERR_TIMEOUT = -7
ERR_GUARD = -8
STATUS_NAMES = {0: "OK", -1: "INVALID", -2: "ALIGN", -3: "NONFINITE", -4: "NOT_CONVERGED",
                -5: "CUDA", -6: "OOM", -7: "TIMEOUT", -8: "GUARD"}
_HARD_ERRORS = {ERR_INVALID, ERR_ALIGN, ERR_CUDA, ERR_OOM}


class IsolocoError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{STATUS_NAMES.get(code, code)}: {msg}")
        self.code = code


class Param(ctypes.Structure):
    _fields_ = [("offset", ctypes.c_int64), ("rows", ctypes.c_int32), ("cols", ctypes.c_int32)]


class Opts(ctypes.Structure):
    _fields_ = [("alpha", ctypes.c_float), ("outer_lr", ctypes.c_float), ("momentum", ctypes.c_float),
                ("reduce_mean", ctypes.c_int), ("max_iter", ctypes.c_int), ("tol", ctypes.c_float),
                ("sync", ctypes.c_int), ("fast_steps", ctypes.c_int), ("orth_target", ctypes.c_int),
                ("momentum_kind", ctypes.c_int), ("scale_kind", ctypes.c_int), ("aggregator", ctypes.c_int),
                ("sparsity", ctypes.c_float), ("seed", ctypes.c_uint), ("spectrum_kind", ctypes.c_int),
                ("full_precision", ctypes.c_int), ("precision_schedule", ctypes.c_longlong)]


_lib = None
_lock = threading.Lock()
_vp = ctypes.c_void_p


def lib():
    """Loads (building first if needed) the CUDA library; raises if that fails."""
    global _lib
    with _lock:
        if _lib is None:
            path = _build.build()
            L = ctypes.CDLL(path)
            L.isoloco_last_error.restype = ctypes.c_char_p
            L.isoloco_opts_default.argtypes = [ctypes.POINTER(Opts)]
            L.isoloco_plan_create.argtypes = [ctypes.POINTER(_vp), ctypes.POINTER(Param), ctypes.c_int,
                                              ctypes.c_int64, ctypes.c_int, ctypes.c_int]
            L.isoloco_plan_destroy.argtypes = [_vp]
            L.isoloco_plan_destroy.restype = None
            L.isoloco_plan_workspace_bytes.argtypes = [_vp]
            L.isoloco_plan_workspace_bytes.restype = ctypes.c_int64
            L.isoloco_plan_num_matrices.argtypes = [_vp]
            L.isoloco_outer_step.argtypes = [_vp, _vp, _vp, ctypes.POINTER(_vp), ctypes.POINTER(Opts), _vp, _vp]
            L.isoloco_outer_step_host.argtypes = [_vp, _vp, _vp, ctypes.POINTER(_vp), ctypes.POINTER(Opts), _vp]
            L.diloco_outer_step.argtypes = [_vp, _vp, _vp, ctypes.POINTER(_vp), ctypes.POINTER(Opts), _vp]
            L.iso_c_merge.argtypes = [_vp, _vp, ctypes.POINTER(_vp), ctypes.c_float, _vp, _vp]
            L.isoloco_last_status.argtypes = [_vp, _vp]
            L.isoloco_read_diag.argtypes = [_vp, _vp, _vp, _vp, _vp, _vp]
            L.isoloco_read_singular_values.argtypes = [_vp, _vp, ctypes.c_int, _vp, ctypes.c_int]
            L.isoloco_check_guards.argtypes = [_vp, _vp]
            L.isoloco_debug_touch_guard.argtypes = [_vp, ctypes.c_int, ctypes.c_int]
            L.isoloco_profile_enable.argtypes = [_vp, ctypes.c_int]
            L.isoloco_profile_read.argtypes = [_vp, _vp, _vp, _vp, ctypes.c_int]
            L.isoloco_plan_launches.argtypes = [_vp]
            L.isoloco_plan_launches.restype = ctypes.c_int64
            L.isoloco_debug_gemm.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                             ctypes.c_int, ctypes.c_int, _vp, _vp, _vp, _vp]
            L.isoloco_debug_gemm_noalloc.argtypes = L.isoloco_debug_gemm.argtypes
            L.isoloco_debug_wait_timeout.argtypes = [ctypes.c_int64, ctypes.POINTER(ctypes.c_int64), _vp]
            _lib = L
    return _lib


def library_path() -> str:
    return _build.LIB


def last_error() -> str:
    return lib().isoloco_last_error().decode(errors="replace")


def _check(rc: int, what: str, hard_only: bool = True) -> int:
    if rc != OK and (rc in _HARD_ERRORS or not hard_only):
        raise IsolocoError(rc, f"{what}: {last_error()}")
    return rc


def _stream(stream=None) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream) if hasattr(stream, "cuda_stream") else int(stream or 0)


def make_opts(alpha=1.0, outer_lr=0.7, momentum=0.9, reduce_mean=True, max_iter=0, tol=0.0,
              sync=False, fast_steps=0, orth_target=0, momentum_kind=0, scale_kind=0, aggregator=0,
              sparsity=0.0, seed=0, spectrum_kind=0, full_precision=0, precision_schedule=0) -> Opts:
    """Options of an outer step; fast_steps > 0 selects the fixed-step variant of Sec. 4.3,
    orth_target / momentum_kind / scale_kind / spectrum_kind (1 clip_high, 2 clip_low, 3 Iso-C
    from the exact singular values) the
    ablations of Sec. 4.5 / App. B, and aggregator / sparsity / seed the merging rule of
    diloco_outer_step (Sec. 3.2: 0 mean, 1 TIES, 2 DARE); full_precision = 1 splits both
    operands of every polar step; see include/isoloco.h."""
    o = Opts()
    lib().isoloco_opts_default(ctypes.byref(o))
    o.alpha, o.outer_lr, o.momentum = float(alpha), float(outer_lr), float(momentum)
    o.reduce_mean, o.max_iter, o.tol, o.sync = int(bool(reduce_mean)), int(max_iter), float(tol), int(bool(sync))
    o.fast_steps = int(fast_steps)
    o.orth_target, o.momentum_kind, o.scale_kind = int(orth_target), int(momentum_kind), int(scale_kind)
    o.aggregator, o.sparsity, o.seed = int(aggregator), float(sparsity), int(seed) & 0xFFFFFFFF
    o.spectrum_kind = int(spectrum_kind)
    o.full_precision = int(full_precision)
    o.precision_schedule = int(precision_schedule)
    return o


def precision_code(std_gp=(0, 0), std_upd=(0, 0), deep_gp=(0, 0), deep_upd=(0, 0)) -> int:
    """Packs a precision schedule (isoloco_opts_t::precision_schedule): per schedule kind,
    the quintic step ranges [from, to) whose Gram and polynomial, and whose update, run one
    pass."""
    f = list(std_gp) + list(std_upd) + list(deep_gp) + list(deep_upd)
    assert all(0 <= v < 32 for v in f)
    return sum(v << (5 * i) for i, v in enumerate(f))


def _ptr_array(tensors) -> ctypes.Array:
    return (_vp * len(tensors))(*[t.data_ptr() for t in tensors])


def _replica_list(replicas) -> list:
    if isinstance(replicas, torch.Tensor):
        return [replicas[k] for k in range(replicas.shape[0])]
    return list(replicas)


class Plan:
    """A parameter table bound to a workspace on the current CUDA device."""

    def __init__(self, table: Sequence, n_total: int, K: int, replica_dtype=torch.float32):
        self._L = lib()
        arr = (Param * max(1, len(table)))()
        for i, (off, r, c) in enumerate(table):
            arr[i].offset, arr[i].rows, arr[i].cols = int(off), int(r), int(c)
        self.table = [tuple(int(x) for x in t) for t in table]
        self.n_total, self.K = int(n_total), int(K)
        self.replica_dtype = replica_dtype
        code = 1 if replica_dtype == torch.bfloat16 else 0
        h = _vp()
        _check(self._L.isoloco_plan_create(ctypes.byref(h), arr, len(table), self.n_total, self.K, code),
               "isoloco_plan_create")
        self._h = h

    # -- lifetime
    def close(self):
        if getattr(self, "_h", None):
            self._L.isoloco_plan_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @property
    def workspace_bytes(self) -> int:
        return int(self._L.isoloco_plan_workspace_bytes(self._h))

    @property
    def num_matrices(self) -> int:
        return int(self._L.isoloco_plan_num_matrices(self._h))

    # -- steps
    def _reps(self, replicas):
        reps = _replica_list(replicas)
        if len(reps) != self.K:
            raise ValueError(f"expected {self.K} replicas, got {len(reps)}")
        for r in reps:
            if r.dtype != self.replica_dtype or not r.is_cuda or r.numel() < self.n_total:
                raise ValueError("replica dtype/device/size does not match the plan")
        return reps

    def outer_step(self, theta: torch.Tensor, momentum: torch.Tensor, replicas, opts: Optional[Opts] = None,
                   update_out: Optional[torch.Tensor] = None, stream=None) -> int:
        """IsoLoCo outer step (Alg. 2), in place on theta and momentum."""
        reps = self._reps(replicas)
        arr = _ptr_array(reps)
        o = opts or make_opts()
        rc = self._L.isoloco_outer_step(self._h, theta.data_ptr(), momentum.data_ptr(), arr, ctypes.byref(o),
                                        _stream(stream), update_out.data_ptr() if update_out is not None else None)
        return _check(rc, "isoloco_outer_step")

    def outer_step_host(self, theta, momentum, replicas, opts: Optional[Opts] = None, stream=None) -> int:
        """Same step on host (CPU, ideally pinned) tensors; copies happen inside the call."""
        reps = _replica_list(replicas)
        arr = _ptr_array(reps)
        o = opts or make_opts()
        rc = self._L.isoloco_outer_step_host(self._h, theta.data_ptr(), momentum.data_ptr(), arr, ctypes.byref(o),
                                             _stream(stream))
        return _check(rc, "isoloco_outer_step_host")

    def diloco_outer_step(self, theta, momentum, replicas, opts: Optional[Opts] = None, stream=None) -> int:
        """DiLoCo outer step (Alg. 1, Nesterov SGD), in place."""
        reps = self._reps(replicas)
        arr = _ptr_array(reps)
        o = opts or make_opts()
        rc = self._L.diloco_outer_step(self._h, theta.data_ptr(), momentum.data_ptr(), arr, ctypes.byref(o),
                                       _stream(stream))
        return _check(rc, "diloco_outer_step")

    def iso_c_merge(self, base, experts, alpha: float, out, stream=None) -> int:
        """Iso-C merge of the plan's K experts into base; result in out."""
        reps = self._reps(experts)
        arr = _ptr_array(reps)
        rc = self._L.iso_c_merge(self._h, base.data_ptr(), arr, float(alpha), out.data_ptr(), _stream(stream))
        return _check(rc, "iso_c_merge")

    def last_status(self, stream=None) -> int:
        return int(self._L.isoloco_last_status(self._h, _stream(stream)))

    def profile(self, enable: bool = True):
        """Turns per-phase CUDA-event timing on or off (resets the accumulators)."""
        _check(self._L.isoloco_profile_enable(self._h, int(bool(enable))), "isoloco_profile_enable")

    def profile_read(self, stream=None):
        """{phase: (milliseconds, launches)} accumulated since profile() was called."""
        n = len(PHASES)
        ms = (ctypes.c_double * n)()
        cnt = (ctypes.c_int64 * n)()
        _check(self._L.isoloco_profile_read(self._h, _stream(stream), ms, cnt, n), "isoloco_profile_read")
        return {ph: (ms[i], cnt[i]) for i, ph in enumerate(PHASES)}

    @property
    def launches(self) -> int:
        """Kernels launched by this plan since its creation."""
        return int(self._L.isoloco_plan_launches(self._h))

    def read_diag(self, stream=None):
        n = self.num_matrices
        sb = (ctypes.c_float * max(1, n))()
        it = (ctypes.c_int32 * max(1, n))()
        st = (ctypes.c_int32 * max(1, n))()
        rs = (ctypes.c_float * max(1, n))()
        _check(self._L.isoloco_read_diag(self._h, _stream(stream), sb, it, st, rs), "isoloco_read_diag")
        return {"sigma_bar": list(sb)[:n], "iters": list(it)[:n], "status": list(st)[:n],
                "residual": list(rs)[:n]}

    def check_guards(self, stream=None) -> int:
        """Compares the guard bytes around every workspace region (isoloco_check_guards):
        0, or ERR_GUARD with last_error() naming the region."""
        return self._L.isoloco_check_guards(self._h, _stream(stream))

    def singular_values(self, matrix: int, stream=None) -> list:
        """Descending singular values of 2-D tensor `matrix` (table order over the 2-D
        tensors) from the last step with spectrum_kind = 3."""
        cap = 1 << 16
        buf = (ctypes.c_float * cap)()
        n = self._L.isoloco_read_singular_values(self._h, _stream(stream), int(matrix), buf, cap)
        if n < 0:
            _check(n, "isoloco_read_singular_values")
        return list(buf)[:n]


def debug_gemm(A: torch.Tensor, B: torch.Tensor, a_mn_major: bool, b_mn_major: bool, M: int, N: int, K: int,
               precision: int = 0, stream=None) -> torch.Tensor:
    """Split-precision tcgen05 GEMM: D[b] = op(A[b]) op(B[b]) (see include/isoloco.h)."""
    batch = A.shape[0]
    D = torch.empty((batch, M, N), dtype=torch.float32, device=A.device)
    rc = lib().isoloco_debug_gemm(int(a_mn_major), int(b_mn_major), int(precision), batch, M, N, K, A.data_ptr(),
                                  B.data_ptr(), D.data_ptr(), _stream(stream))
    _check(rc, "isoloco_debug_gemm", hard_only=False)
    return D


def debug_gemm_noalloc(A: torch.Tensor, B: torch.Tensor, D: torch.Tensor, a_mn_major: bool, b_mn_major: bool,
                       M: int, N: int, K: int, precision: int = 0, stream=None) -> int:
    """The same GEMM as debug_gemm into the caller's D, with the library's static scratch
    (no device allocation; see isoloco_debug_gemm_noalloc in include/isoloco.h)."""
    if D.dtype != torch.float32 or D.numel() < A.shape[0] * M * N:
        raise ValueError("D must be fp32 with room for batch x M x N")
    rc = lib().isoloco_debug_gemm_noalloc(int(a_mn_major), int(b_mn_major), int(precision), A.shape[0], M, N, K,
                                          A.data_ptr(), B.data_ptr(), D.data_ptr(), _stream(stream))
    return _check(rc, "isoloco_debug_gemm_noalloc", hard_only=False)


def debug_wait_timeout(limit_ns: int, stream=None):
    """A bounded device wait that nothing ends runs out after limit_ns (see
    isoloco_debug_wait_timeout in include/isoloco.h).  Returns (status, elapsed_ns)."""
    el = ctypes.c_int64(0)
    rc = lib().isoloco_debug_wait_timeout(int(limit_ns), ctypes.byref(el), _stream(stream))
    if rc not in (OK, ERR_TIMEOUT):
        raise IsolocoError(rc, f"isoloco_debug_wait_timeout: {last_error()}")
    return rc, el.value
