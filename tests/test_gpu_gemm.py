"""The tcgen05 GEMM entry point (ld_gemm_bf16) against a float64 matmul of
the same bf16 operands, for every operand-major combination, ragged M and N
tiles, the empty contraction and both output types."""

import pytest
import torch

import paper_2609_05275_gb300 as P

pytestmark = pytest.mark.gpu


def _operands(M, N, K, a_mn, b_mn, seed):
    g = torch.Generator(device="cpu").manual_seed(seed)
    A = torch.randn((M, K), generator=g).to(torch.bfloat16)
    B = torch.randn((N, K), generator=g).to(torch.bfloat16)
    Ad = (A.t().contiguous() if a_mn else A).cuda()
    Bd = (B.t().contiguous() if b_mn else B).cuda()
    ref = A.double() @ B.double().t()
    return Ad, Bd, ref


@pytest.mark.parametrize("a_mn,b_mn", [(0, 0), (0, 1), (1, 0), (1, 1)])
@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (256, 512, 320), (192, 384, 128), (64, 128, 64),
                                   (640, 1280, 1024), (384, 6144 // 16, 512)])
def test_gemm_matches_float64(M, N, K, a_mn, b_mn):
    Ad, Bd, ref = _operands(M, N, K, a_mn, b_mn, seed=M * 7 + N + K)
    lda = M if a_mn else K
    ldb = N if b_mn else K
    for out_dtype in (torch.float32, torch.bfloat16):
        D = torch.full((M, N), float("nan"), device="cuda", dtype=out_dtype)
        P.ld_gemm_bf16(M, N, K, Ad, lda, a_mn, Bd, ldb, b_mn, D, N, alpha=0.5)
        torch.cuda.synchronize()
        got = D.double().cpu()
        err = (got - 0.5 * ref).abs().max().item()
        scale = (0.5 * ref).abs().max().item()
        tol = 1e-5 * scale + 1e-5 if out_dtype == torch.float32 else 8e-3 * scale
        assert err <= tol, (out_dtype, err, tol)


def test_gemm_empty_contraction_writes_zero():
    M, N = 128, 256
    A = torch.zeros((M, 64), device="cuda", dtype=torch.bfloat16)
    B = torch.zeros((N, 64), device="cuda", dtype=torch.bfloat16)
    D = torch.full((M, N), 7.0, device="cuda", dtype=torch.float32)
    P.ld_gemm_bf16(M, N, 0, A, 64, 0, B, 64, 0, D, N)
    torch.cuda.synchronize()
    assert (D == 0).all()


def test_gemm_status_word_untouched_and_strided_output():
    M, N, K = 256, 256, 256
    Ad, Bd, ref = _operands(M, N, K, 0, 0, seed=5)
    status = torch.zeros(4, dtype=torch.int32, device="cuda")
    D = torch.zeros((M, N + 64), device="cuda", dtype=torch.float32)
    P.ld_gemm_bf16(M, N, K, Ad, K, 0, Bd, K, 0, D, N + 64, status=status)
    torch.cuda.synchronize()
    assert int(status[0]) == 0
    assert (D[:, N:] == 0).all()
    assert (D[:, :N].double().cpu() - ref).abs().max().item() <= 1e-5 * ref.abs().max().item() + 1e-5
