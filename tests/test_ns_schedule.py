"""The polynomial schedules compiled into the library (csrc/ns_schedule.h), checked on the CPU.

Each step is an odd quintic p(x) = a x + b x^3 + c x^5 applied to every singular value
of the iterate.  What the polar iteration relies on, checked here by evaluating the
coefficients exactly as compiled:
  * p(x) > 0 wherever a singular value can be (no direction collapses or changes sign,
    which would converge to a different orthogonal factor), with the 0.2 x cushion;
  * composing the steps maps every value in [ell, 1] into [0.998, 1.002] (the interval
    the convergence test and the cubic polish then finish from);
  * tiny values grow by the product of the linear coefficients;
  * the header matches what the generator produces now.
"""
import os
import re

import numpy as np
import pytest

HEADER = os.path.join(os.path.dirname(__file__), "..", "paper_2607_03011_gb300", "csrc", "ns_schedule.h")


def compiled(name):
    txt = open(HEADER).read()
    blk = txt.split(f"static __constant__ float {name}[")[1].split("};")[0]
    rows = re.findall(r"\{([-0-9.e]+)f, ([-0-9.e]+)f, ([-0-9.e]+)f\}", blk)
    # as the GPU sees them: fp32 constants
    return [tuple(np.float32(float(v)) for v in r) for r in rows]


SCHEDULES = [("kSched", 1e-3, 7), ("kSchedDeep", 1e-6, 12)]


@pytest.mark.parametrize("name,ell,steps", SCHEDULES)
def test_steps_keep_every_singular_value_positive(name, ell, steps):
    sched = compiled(name)
    assert len(sched) == steps
    xs = np.concatenate([np.geomspace(1e-9, 1.0, 20001), np.linspace(1e-6, 2.01, 20001)])
    for a, b, c in sched:
        ratio = float(a) + float(b) * xs ** 2 + float(c) * xs ** 4   # p(x) / x
        assert ratio.min() >= 0.2 - 1e-4


@pytest.mark.parametrize("name,ell,steps", SCHEDULES)
def test_composition_maps_the_design_interval_to_one(name, ell, steps):
    sched = compiled(name)
    x = np.concatenate([np.geomspace(ell, 1.0, 50001), np.linspace(ell, 1.02, 50001)])
    for a, b, c in sched:
        x = float(a) * x + float(b) * x ** 3 + float(c) * x ** 5
    assert x.min() >= 0.998 - 1e-6 and x.max() <= 1.002 + 1e-6


@pytest.mark.parametrize("name,ell,steps", SCHEDULES)
def test_tiny_values_grow_by_the_linear_coefficients(name, ell, steps):
    sched = compiled(name)
    x0 = ell * 1e-3
    x = x0
    for a, b, c in sched:
        x = float(a) * x + float(b) * x ** 3 + float(c) * x ** 5
    assert x == pytest.approx(x0 * np.prod([float(a) for a, _, _ in sched]), rel=1e-3)


def test_header_is_what_the_generator_writes(tmp_path):
    pytest.importorskip("scipy")
    from paper_2607_03011_gb300 import ns_schedule
    out = tmp_path / "ns_schedule.h"
    ns_schedule.write_header(str(out))
    assert out.read_text() == open(HEADER).read()
