"""Split-precision tcgen05 GEMM (the building block of the polar iteration) vs fp64.

Covers the three operand-layout pairs the polar iteration uses (K/K for G^2 and
the tall update, MN/MN for the tall Gram, K/MN for the wide update) on tiles that
are full, ragged, and smaller than one tile, with several batch entries.
Tolerance: ~2^-16 per operand from the bf16 hi+lo split -> relative Frobenius
error <= 3e-5 against fp64; a single bf16 pass would be ~2e-3.
"""
import pytest
import torch

pytestmark = pytest.mark.gpu

CASES = [
    (2, 128, 256, 64),
    (3, 256, 512, 1024),
    (2, 65, 130, 70),
    (1, 1, 1, 1),
    (2, 300, 40, 999),
    (1, 1024, 1024, 2816),
]


@pytest.fixture(scope="module")
def iso():
    from paper_2607_03011_gb300 import isoloco
    isoloco.lib()
    return isoloco


def _ref(A, B, a_mn, b_mn):
    Ad = A.double().transpose(1, 2) if a_mn else A.double()     # [b, M, K]
    Bd = B.double().transpose(1, 2) if b_mn else B.double()     # [b, N, K]
    return Ad @ Bd.transpose(1, 2)


@pytest.mark.parametrize("a_mn,b_mn", [(0, 0), (1, 1), (0, 1), (1, 0)])
@pytest.mark.parametrize("batch,M,N,K", CASES)
def test_debug_gemm_layouts(iso, a_mn, b_mn, batch, M, N, K):
    g = torch.Generator(device="cuda").manual_seed(M * 7 + N * 3 + K)
    A = torch.randn((batch, K, M) if a_mn else (batch, M, K), device="cuda", generator=g)
    B = torch.randn((batch, K, N) if b_mn else (batch, N, K), device="cuda", generator=g)
    D = iso.debug_gemm(A, B, a_mn, b_mn, M, N, K)
    R = _ref(A, B, a_mn, b_mn)
    err = (D.double() - R).norm() / R.norm()
    assert err < 3e-5, float(err)
    # the split is what buys the accuracy: one bf16 pass is ~100x worse
    one_pass = _ref(A.bfloat16().float(), B.bfloat16().float(), a_mn, b_mn)
    if K >= 16:
        assert (one_pass - R).norm() / R.norm() > 10 * err


# precision 1: fp16, A split / B single; 2: A single / B split; 3: both split.
# Expected relative error: the single operand's fp16 rounding (2^-12 relative per
# entry, ~1.4e-4 in Frobenius norm on random data) for 1 and 2; for 3 the fp32
# accumulation over long K dominates (~1e-5 at K = 2816, below bf16's 3e-5).
@pytest.mark.parametrize("precision,tol", [(1, 4e-4), (2, 4e-4), (3, 2e-5)])
@pytest.mark.parametrize("a_mn,b_mn", [(0, 0), (1, 1), (0, 1)])
@pytest.mark.parametrize("batch,M,N,K", [(2, 128, 256, 64), (2, 65, 130, 70), (1, 1024, 1024, 2816)])
def test_debug_gemm_fp16_passes(iso, precision, tol, a_mn, b_mn, batch, M, N, K):
    g = torch.Generator(device="cuda").manual_seed(M + N + K + precision)
    A = torch.randn((batch, K, M) if a_mn else (batch, M, K), device="cuda", generator=g)
    B = torch.randn((batch, K, N) if b_mn else (batch, N, K), device="cuda", generator=g)
    D = iso.debug_gemm(A, B, a_mn, b_mn, M, N, K, precision=precision)
    R = _ref(A, B, a_mn, b_mn)
    err = float((D.double() - R).norm() / R.norm())
    assert err < tol, err
    if precision in (1, 2):
        # matches the model: only the single operand is rounded to fp16
        A1 = A if precision == 1 else A.half().float()
        B1 = B if precision == 2 else B.half().float()
        model = _ref(A1, B1, a_mn, b_mn)
        assert float((D.double() - model).norm() / R.norm()) < 0.1 * err


def test_debug_gemm_deterministic(iso):
    g = torch.Generator(device="cuda").manual_seed(5)
    A = torch.randn((2, 256, 512), device="cuda", generator=g)
    B = torch.randn((2, 512, 512), device="cuda", generator=g)
    D1 = iso.debug_gemm(A, B, 0, 1, 256, 512, 512)
    D2 = iso.debug_gemm(A, B, 0, 1, 256, 512, 512)
    assert torch.equal(D1, D2)


def test_bounded_wait_runs_out_and_the_context_survives(iso):
    """The pipeline's bounded mbarrier wait on a barrier that nothing arrives on gives up
    after its limit and reports TIMEOUT; the GPU context stays usable (a GEMM right after
    is exact).  Limits outside 1 ms .. 1 s are refused before any launch."""
    rc, elapsed = iso.debug_wait_timeout(20_000_000)
    assert rc == iso.ERR_TIMEOUT
    assert 20_000_000 <= elapsed < 1_000_000_000
    with pytest.raises(iso.IsolocoError):
        iso.debug_wait_timeout(1_000)
    with pytest.raises(iso.IsolocoError):
        iso.debug_wait_timeout(2_000_000_000)
    g = torch.Generator(device="cuda").manual_seed(9)
    A = torch.randn((1, 256, 512), device="cuda", generator=g)
    B = torch.randn((1, 256, 512), device="cuda", generator=g)
    D = iso.debug_gemm(A, B, 0, 0, 256, 256, 512)
    ref = _ref(A, B, 0, 0)
    assert ((D.double() - ref).norm() / ref.norm()).item() < 3e-5
