"""The failure path of the pipelined kernels, exercised without a fault: a
bounded wait that nothing completes gives up after its limit, records
LD_ERR_TIMEOUT in the status word, and the context stays usable (a GEMM
launched afterwards is correct)."""

import time

import pytest
import torch

import paper_2609_05275_gb300 as P

pytestmark = pytest.mark.gpu


def test_bounded_wait_records_timeout_and_context_survives():
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    P.ld_check_wait_timeout(status)
    torch.cuda.synchronize()
    waited = time.perf_counter() - t0
    assert int(status.item()) == P.LD_ERR_TIMEOUT
    assert 1.0 < waited < 30.0
    # an earlier nonzero status is kept
    status.fill_(P.LD_ERR_CUDA)
    P.ld_check_wait_timeout(status)
    torch.cuda.synchronize()
    assert int(status.item()) == P.LD_ERR_CUDA
    # the context still runs work correctly
    g = torch.Generator(device="cpu").manual_seed(0)
    A = torch.randn(128, 64, generator=g).to("cuda", torch.bfloat16)
    B = torch.randn(128, 64, generator=g).to("cuda", torch.bfloat16)
    D = torch.empty(128, 128, device="cuda", dtype=torch.float32)
    s2 = torch.zeros(1, dtype=torch.int32, device="cuda")
    P.ld_gemm_bf16(128, 128, 64, A, 64, 0, B, 64, 0, D, 128, status=s2)
    torch.cuda.synchronize()
    ref = A.float() @ B.float().t()
    assert int(s2.item()) == 0
    assert torch.allclose(D, ref, rtol=1e-3, atol=1e-3)
