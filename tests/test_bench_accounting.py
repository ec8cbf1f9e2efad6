"""The benchmark's roofline accounting (CPU): output tiles, executed and algorithmic FLOPs of
the polar GEMMs, and the streaming kernels' bytes, against counts worked out by hand."""
import os
import re
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_tile_constants_match_the_kernel():
    """bench's tile is the CTA pair's 256 x 256 output tile, 64 deep, as the kernel defines it."""
    src = open(os.path.join(ROOT, "paper_2607_03011_gb300", "csrc", "types.h")).read()
    val = {k: int(v) for k, v in re.findall(r"constexpr int (BM|BN|BK) = (\d+);", src)}
    assert "kTileM = kPairMma ? 2 * BM : BM" in src and "constexpr bool kPairMma = true" in src
    assert (bench.BM, bench.BN, bench.BK) == (2 * val["BM"], val["BN"], val["BK"])


@pytest.mark.parametrize("n, tiles", [(1, 1), (64, 1), (256, 1), (257, 3), (512, 3), (1024, 10), (1025, 15)])
def test_sym_tiles(n, tiles):
    """Tiles on or above the diagonal of a ceil(n / 256)-square tile grid: T (T + 1) / 2."""
    assert bench._sym_tiles(n) == tiles
    t = -(-n // 256)
    assert sum(1 for tm in range(t) for tn in range(t) if tn >= tm) == tiles


def _diag(iters, status=None):
    return {"iters": list(iters), "status": list(status or [0] * len(iters))}


def test_algorithmic_flops_square():
    """A converged 1024 x 1024 matrix after 12 iterations: 12 Grams and updates (2 n^3 each),
    11 quintic G^2 products (the last iteration is the cubic polish)."""
    n = 1024
    fl = bench.gemm_flops([("w", n, n)], _diag([12]))
    assert fl == {"gram": 12 * 2.0 * n ** 3, "poly": 11 * 2.0 * n ** 3, "update": 12 * 2.0 * n ** 3}
    # not converged (max_iter reached): one more Gram (the failed test), every step quintic
    fl = bench.gemm_flops([("w", n, n)], _diag([12], [1]))
    assert fl == {"gram": 13 * 2.0 * n ** 3, "poly": 12 * 2.0 * n ** 3, "update": 12 * 2.0 * n ** 3}


def test_algorithmic_flops_rectangular_and_1d():
    """A 2816 x 1024 matrix: Gram and update 2 * 2816 * 1024^2 each, G^2 2 * 1024^3; 1-D
    tensors cost nothing."""
    fl = bench.gemm_flops([("v", 7, 0), ("w", 2816, 1024)], _diag([7]))
    assert fl["gram"] == 7 * 2.0 * 2816 * 1024 ** 2
    assert fl["update"] == 7 * 2.0 * 2816 * 1024 ** 2
    assert fl["poly"] == 6 * 2.0 * 1024 ** 3


def test_executed_flops_square():
    """1024 x 1024, 12 iterations, converged.  One Gram or G^2 pass over the 10 upper tiles:
    10 * 256 * 256 * 2 * 1024; one update pass over all 16 tiles: 16 * 256 * 256 * 2 * 1024.
    Iteration 0 and the polish update take three passes, the rest two; with `full` three."""
    g1 = 10 * 256 * 256 * 2.0 * 1024
    u1 = 16 * 256 * 256 * 2.0 * 1024
    fx = bench.gemm_exec_flops([("w", 1024, 1024)], _diag([12]), sched=bench.NO_DEMOTION)
    assert fx == {"gram": (3 + 2 * 11) * g1, "poly": (3 + 2 * 10) * g1, "update": (3 + 3 + 2 * 10) * u1}
    # the default schedule: a 1024 x 1024 matrix is near-square (deep schedule, quintic steps
    # 0 .. 10): Grams leading to steps 9, 10 and G^2 of steps 9, 10 single-pass, the update of
    # step 10 too
    fx = bench.gemm_exec_flops([("w", 1024, 1024)], _diag([12]))
    assert fx == {"gram": (3 + 2 * 9 + 1 * 2) * g1, "poly": (3 + 2 * 8 + 1 * 2) * g1,
                  "update": (3 + 2 * 9 + 1 + 3) * u1}
    fx = bench.gemm_exec_flops([("w", 1024, 1024)], _diag([12]), full=True)
    assert fx == {"gram": 36 * g1, "poly": 33 * g1, "update": 36 * u1}
    fx = bench.gemm_exec_flops([("w", 1024, 1024)], _diag([5]), fast=True)
    assert fx == {"gram": 15 * g1, "poly": 15 * g1, "update": 15 * u1}


def test_executed_flops_ragged_padding():
    """300 x 257: n = 257 pads to 320 (five 64-deep k-blocks), the long side to 320; the
    update covers 2 x 2 tiles of 256, the symmetric products 3 tiles."""
    g1 = 3 * 256 * 256 * 2.0 * 320
    p1 = 3 * 256 * 256 * 2.0 * 320
    u1 = 4 * 256 * 256 * 2.0 * 320
    fx = bench.gemm_exec_flops([("w", 300, 257)], _diag([1]))
    # one iteration: iteration 0 is also the polish (three passes, no G^2)
    assert fx == {"gram": 3 * g1, "poly": 0.0, "update": 3 * u1}
    fx = bench.gemm_exec_flops([("w", 300, 257)], _diag([2]), sched=bench.NO_DEMOTION)
    assert fx == {"gram": (3 + 2) * g1, "poly": 3 * p1, "update": 6 * u1}
    # default schedule (standard kind): the Gram of iteration 1 leads to step 1, single-pass
    fx = bench.gemm_exec_flops([("w", 300, 257)], _diag([2]))
    assert fx == {"gram": (3 + 1) * g1, "poly": 3 * p1, "update": 6 * u1}


def test_executed_flops_standard_schedule_default():
    """2816 x 1024 (standard schedule), 7 iterations: quintic steps 0 .. 5, polish at 6.
    Grams leading to steps 1 .. 5 and G^2 of steps 1 .. 5 single-pass (the Gram before the
    polish keeps two), updates of steps 2 .. 5 single-pass, step 1's two, the polish three."""
    n, m = 1024, 2816
    kp = 2816  # 2816 = 44 k-blocks of 64
    g1 = 10 * 256 * 256 * 2.0 * kp
    p1 = 10 * 256 * 256 * 2.0 * 1024
    u1 = 11 * 4 * 256 * 256 * 2.0 * 1024
    fx = bench.gemm_exec_flops([("w", m, n)], _diag([7]))
    assert fx == {"gram": (3 + 5 * 1 + 2) * g1, "poly": (3 + 5 * 1) * p1, "update": (3 + 2 + 4 * 1 + 3) * u1}


def test_default_schedule_matches_the_library():
    """bench's mirror of the default precision schedule is the library's constant."""
    src = open(os.path.join(ROOT, "paper_2607_03011_gb300", "csrc", "api.cu")).read()
    body = src.split("constexpr long long kDefaultPrecisionSchedule =")[1].split(";")[0]
    fields = [int(v) for v, _ in re.findall(r"\((\d+)ll << (\d+)\)", body)]
    d = bench.DEFAULT_SCHEDULE
    assert fields == [d["std"]["gp"][0], d["std"]["gp"][1], d["std"]["upd"][0], d["std"]["upd"][1],
                      d["deep"]["gp"][0], d["deep"]["gp"][1], d["deep"]["upd"][0], d["deep"]["upd"][1]]


def test_stream_bytes():
    """Per parameter: the reduce reads K replicas and theta and writes 4 bytes of Delta; the
    apply reads theta, B and an 8-byte U source and writes theta and B; the trace reads Q and
    Delta planes (8 bytes per matrix element)."""
    table = [("a", 4, 3), ("b", 5, 0)]      # 12 matrix elements, 17 parameters
    sb = bench.stream_bytes(table, K=8, replica_bytes=4)
    assert sb == {"reduce": 36 * 17 + 4 * 17, "apply": 20 * 17, "trace": 8 * 12,
                  "algorithmic_step": 48 * 17 + 8 * 12}
    sb = bench.stream_bytes(table, K=4, replica_bytes=2)
    assert sb["reduce"] == (4 * 2 + 4) * 17 + 4 * 17


def test_gram_side_rule_matches_the_library():
    """bench's Gram-side rule (rows >= ratio * cols, rows >= 2 k-blocks) is the library's."""
    src = open(os.path.join(ROOT, "paper_2607_03011_gb300", "csrc", "types.h")).read()
    assert int(re.search(r"constexpr int kGramSideRatio = (\d+);", src).group(1)) == bench.GRAM_SIDE_RATIO
    api = open(os.path.join(ROOT, "paper_2607_03011_gb300", "csrc", "api.cu")).read()
    assert "bk.tall && t.rows >= kGramSideRatio * t.cols && t.rows >= 2 * BK" in api
    assert bench.gram_side(32000, 1024) and not bench.gram_side(2816, 1024) and not bench.gram_side(1024, 1024)
    assert not bench.gram_side(32000, 1024, full=True) and not bench.gram_side(32000, 1024, fast=True)


def test_algorithmic_flops_gram_side():
    """32000 x 1024, 7 iterations, converged (quintic steps 0 .. 5, polish at 6): iteration 0's
    Gram 2 m n^2 and six more Grams on the n x n side (W = A Z and G = Z^T W, 2 n^3 each),
    six G^2 products, six Z P products and the final Q = Delta Z (2 m n^2)."""
    m, n = 32000, 1024
    fl = bench.gemm_flops([("e", m, n)], _diag([7]))
    assert fl["gram"] == 2.0 * m * n * n + 6 * 2 * 2.0 * n ** 3
    assert fl["poly"] == 6 * 2.0 * n ** 3
    assert fl["update"] == 6 * 2.0 * n ** 3 + 2.0 * m * n * n
    # the same matrix on the full-precision path iterates on the rows x cols side
    fl = bench.gemm_flops([("e", m, n)], _diag([7]), full=True)
    assert fl["update"] == 7 * 2.0 * m * n * n
