"""The RMSNorm-backward step (ld_rmsnorm_backward) against the oracle's
rmsnorm_backward at the Llama-3-8B width (d 4096) on kept rows of several
sequences: the residual-gradient update on exactly the kept rows (others
untouched), the scaled compact copy, and the gain gradient."""

import numpy as np
import pytest
import torch

import paper_2609_05275_gb300 as P
from oracle import stack as OK

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("B,S,d,kept", [(4, 256, 4096, [0, 2, 3]), (3, 64, 128, [1]), (5, 128, 768, [])])
def test_rmsnorm_backward_matches_oracle(B, S, d, kept):
    g = torch.Generator().manual_seed(B * 100 + d)
    M = len(kept) * S
    Mc = max(M, 1)
    dyn = torch.randn(Mc, d, generator=g)
    xs = torch.randn(Mc, d, generator=g)
    gamma = (1 + 0.1 * torch.randn(d, generator=g)).to(torch.bfloat16)
    rstd = (1.0 / torch.sqrt((xs.float() ** 2).mean(dim=1) + 1e-6))
    dx0 = torch.randn(B * S, d, generator=g)
    idx = torch.full((B,), -1, dtype=torch.int32)
    idx[: len(kept)] = torch.tensor(kept, dtype=torch.int32)
    cnt = torch.tensor([len(kept)], dtype=torch.int32)
    dev = lambda t: t.cuda()  # noqa: E731
    ddx = dev(dx0.clone())
    nxt = torch.zeros(Mc, d, dtype=torch.bfloat16, device="cuda")
    dgam = torch.full((d,), float("nan"), device="cuda")
    scratch = torch.empty(P.rmsnorm_backward_scratch_bytes(B, S, d) // 4, device="cuda")
    P.ld_rmsnorm_backward(B, S, d, dev(dyn), dev(xs), dev(rstd), dev(gamma), dev(idx), dev(cnt), ddx, nxt, 1.5,
                          dgam, scratch)
    torch.cuda.synchronize()
    ref_dx = dx0.double().numpy().copy()
    ref_dg = np.zeros(d)
    if M:
        xn = xs.double().numpy() * rstd.double().numpy()[:, None]
        drow, ref_dg = OK.rmsnorm_backward(dyn.double().numpy(), xn, rstd.double().numpy(), gamma.double().numpy())
        rows = np.concatenate([np.arange(b * S, (b + 1) * S) for b in kept])
        ref_dx[rows] += drow
        got_next = nxt.double().cpu().numpy()
        ref_next = 1.5 * ref_dx[rows]
        assert np.abs(got_next - ref_next).max() <= 8e-3 * np.abs(ref_next).max()
    got = ddx.double().cpu().numpy()
    assert np.abs(got - ref_dx).max() <= 1e-5 * np.abs(ref_dx).max()
    untouched = np.ones(B * S, dtype=bool)
    for b in kept:
        untouched[b * S:(b + 1) * S] = False
    assert np.array_equal(got[untouched], dx0.double().numpy()[untouched])
    gd = dgam.double().cpu().numpy()
    assert np.abs(gd - ref_dg).max() <= 1e-5 * max(np.abs(ref_dg).max(), 1.0)
