"""The C-ABI library loads and exports every symbol include/isoloco.h declares.

Runs without a GPU: only argument validation (which returns before any CUDA
call) is exercised here.
"""
import ctypes
import os
import re

import pytest

from conftest import ROOT

HEADER = os.path.join(ROOT, "include", "isoloco.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    body = src[src.index('extern "C"'):]
    names = re.findall(r"^\s*(?:const\s+)?(?:int|void|int64_t|char|isoloco_\w+)\s*\**\s*(\w+)\s*\(", body, flags=re.M)
    return sorted(set(n for n in names if n != "typedef"))


@pytest.fixture(scope="module")
def lib():
    from paper_2607_03011_gb300 import isoloco
    return isoloco.lib()


def test_header_declares_the_entry_points():
    names = declared_functions()
    for n in ["isoloco_plan_create", "isoloco_plan_destroy", "isoloco_outer_step", "diloco_outer_step",
              "iso_c_merge", "isoloco_outer_step_host", "isoloco_last_error", "isoloco_debug_gemm"]:
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_validation_without_gpu(lib):
    from paper_2607_03011_gb300 import isoloco
    o = isoloco.Opts()
    assert lib.isoloco_opts_default(ctypes.byref(o)) == 0
    assert o.alpha == 1.0 and abs(o.outer_lr - 0.7) < 1e-7 and abs(o.momentum - 0.9) < 1e-7
    assert o.reduce_mean == 1 and o.max_iter > 0 and o.tol > 0
    h = ctypes.c_void_p()
    tab = (isoloco.Param * 2)()
    tab[0].offset, tab[0].rows, tab[0].cols = 0, 4, 4
    tab[1].offset, tab[1].rows, tab[1].cols = 8, 4, 0      # overlaps the matrix
    assert lib.isoloco_plan_create(ctypes.byref(h), tab, 2, 100, 2, 0) == isoloco.ERR_INVALID
    assert "overlap" in isoloco.last_error()
    tab[1].offset = 16
    assert lib.isoloco_plan_create(ctypes.byref(h), tab, 2, 100, 0, 0) == isoloco.ERR_INVALID   # K = 0
    assert lib.isoloco_plan_create(ctypes.byref(h), tab, 2, 100, 65, 0) == isoloco.ERR_INVALID  # K > 64
    assert lib.isoloco_plan_create(ctypes.byref(h), tab, 2, 10, 2, 0) == isoloco.ERR_INVALID    # outside n_total
    assert lib.isoloco_plan_create(ctypes.byref(h), tab, 2, 100, 2, 7) == isoloco.ERR_INVALID   # bad dtype
    assert not h.value
    assert lib.isoloco_outer_step(None, None, None, None, None, None, None) == isoloco.ERR_INVALID
    assert lib.diloco_outer_step(None, None, None, None, None, None) == isoloco.ERR_INVALID
    assert lib.isoloco_debug_gemm(0, 0, 0, 0, 1, 1, 1, None, None, None, None) == isoloco.ERR_INVALID
    assert lib.isoloco_debug_gemm(0, 0, 9, 1, 1, 1, 1, None, None, None, None) == isoloco.ERR_INVALID
    assert lib.isoloco_read_singular_values(None, None, 0, None, 0) == isoloco.ERR_INVALID
    assert lib.isoloco_check_guards(None, None) == isoloco.ERR_INVALID
    assert lib.isoloco_debug_wait_timeout(1_000, None, None) == isoloco.ERR_INVALID          # below 1 ms
    assert lib.isoloco_debug_wait_timeout(2_000_000_000, None, None) == isoloco.ERR_INVALID  # above 1 s


def test_opts_layout_matches_the_header(tmp_path, lib):
    """The binding's ctypes mirror of isoloco_opts_t has the header's size and field offsets
    (checked by a C program compiled against include/isoloco.h), and the new fields default
    to the paper's method (mean aggregation, Iso-C spectrum)."""
    import shutil
    import subprocess
    from paper_2607_03011_gb300 import isoloco
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    fields = [f for f, _ in isoloco.Opts._fields_]
    src = tmp_path / "layout.c"
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "isoloco.h"', "int main(void) {",
             '  printf("size %zu\\n", sizeof(isoloco_opts_t));']
    lines += [f'  printf("{f} %zu\\n", offsetof(isoloco_opts_t, {f}));' for f in fields]
    lines += ["  return 0;", "}"]
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    subprocess.run([gcc, "-std=c11", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)], check=True)
    out = dict(line.split() for line in subprocess.run([str(exe)], capture_output=True, text=True,
                                                       check=True).stdout.splitlines())
    assert int(out["size"]) == ctypes.sizeof(isoloco.Opts)
    for f in fields:
        assert int(out[f]) == getattr(isoloco.Opts, f).offset, f
    o = isoloco.Opts()
    assert lib.isoloco_opts_default(ctypes.byref(o)) == 0
    assert (o.fast_steps, o.orth_target, o.momentum_kind, o.scale_kind, o.aggregator, o.sparsity, o.seed,
            o.spectrum_kind, o.full_precision, o.precision_schedule) == (0, 0, 0, 0, 0, 0.0, 0, 0, 0, 0)
