"""ld_rmsnorm_backward_noalloc, the RMSNorm-backward step for callers that
cannot allocate device memory (its scratch is a fixed array inside the
library), against ld_rmsnorm_backward with a caller-provided scratch buffer,
on two calls in a row with different shapes and kept lists: the second call
must not see anything left over from the first.  Kept in its own file so that
pytest collects it last."""

import pytest
import torch

import paper_2609_05275_gb300 as P

pytestmark = pytest.mark.gpu


def _inputs(B, S, d, kept, seed):
    g = torch.Generator().manual_seed(seed)
    M = max(len(kept) * S, 1)
    idx = torch.full((B,), -1, dtype=torch.int32)
    idx[: len(kept)] = torch.tensor(kept, dtype=torch.int32)
    xs = torch.randn(M, d, generator=g)
    return dict(
        dyn=torch.randn(M, d, generator=g).cuda(),
        xs=xs.cuda(),
        rstd=(1.0 / torch.sqrt((xs ** 2).mean(dim=1) + 1e-6)).cuda(),
        gamma=(1 + 0.1 * torch.randn(d, generator=g)).to(torch.bfloat16).cuda(),
        idx=idx.cuda(),
        cnt=torch.tensor([len(kept)], dtype=torch.int32).cuda(),
        dx=torch.randn(B * S, d, generator=g).cuda(),
        M=M,
    )


def _both(B, S, d, kept, seed):
    t = _inputs(B, S, d, kept, seed)
    outs = []
    for noalloc in (False, True):
        dx = t["dx"].clone()
        nxt = torch.zeros(t["M"], d, dtype=torch.bfloat16, device="cuda")
        dg = torch.full((d,), float("nan"), device="cuda")
        args = (B, S, d, t["dyn"], t["xs"], t["rstd"], t["gamma"], t["idx"], t["cnt"], dx, nxt, 0.75, dg)
        if noalloc:
            P.ld_rmsnorm_backward_noalloc(*args)
        else:
            scratch = torch.empty(P.rmsnorm_backward_scratch_bytes(B, S, d) // 4, device="cuda")
            P.ld_rmsnorm_backward(*args, scratch)
        torch.cuda.synchronize()
        outs.append((dx, nxt.float(), dg))
    return outs


def _close(a, b):
    return (a - b).abs().max().item() <= 1e-5 * b.abs().max().item() + 1e-6


def test_noalloc_matches_scratch_entry_point_twice():
    # first call: many blocks at a large width; second: fewer blocks, other
    # kept list, other width
    for B, S, d, kept, seed in ((4, 512, 2048, [0, 1, 3], 1), (3, 128, 768, [2], 2)):
        (dx, nx, dg), (dx2, nx2, dg2) = _both(B, S, d, kept, seed)
        assert _close(dx2, dx) and _close(nx2, nx) and _close(dg2, dg)
        assert torch.isfinite(dg2).all()


def test_noalloc_wide_rows_after_a_larger_call():
    # d > 8192 runs the shared-memory row kernel (its own launch attribute);
    # B*S = 512 gives 64 partial-sum rows of 16384, inside the fixed array.
    # The first call fills more of the array (320 rows at d = 8192), so stale
    # partial sums would show up in the second call's dgamma.
    for B, S, d, kept, seed in ((2, 2048, 8192, [0, 1], 4), (2, 256, 16384, [1, 0], 5)):
        (dx, nx, dg), (dx2, nx2, dg2) = _both(B, S, d, kept, seed)
        assert _close(dx2, dx) and _close(nx2, nx) and _close(dg2, dg)
        assert torch.isfinite(dg2).all()


def test_noalloc_rejects_sizes_beyond_its_array():
    t = _inputs(1, 2560, 16384, [0], 3)
    dg = torch.empty(16384, device="cuda")
    with pytest.raises(P.LdError) as e:
        P.ld_rmsnorm_backward_noalloc(1, 2560, 16384, t["dyn"], t["xs"], t["rstd"], t["gamma"], t["idx"], t["cnt"],
                                      t["dx"], None, 1.0, dg)
    assert e.value.status == P.LD_ERR_SHAPE
