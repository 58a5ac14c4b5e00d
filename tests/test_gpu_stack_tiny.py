"""Forward and backward of the whole stack through the C ABI against the
oracle on the tiny workload (2 layers, d 128, 8 x 64 tokens, p = [0, 0.5])
on the full tensors, for the bf16 tensor-core path and the float32 debug
path; plus the exact special cases p = 1 (identity) and p = 0."""

import numpy as np
import pytest
import torch

from paper_2609_05275_gb300 import synth
from parity import check_close, gpu_run, oracle_run, to_np
from oracle import masks as OM

pytestmark = pytest.mark.gpu


def _inputs(cfg, dtype, gamma_noise=0.0, seed=0):
    host = synth.stack_weights(cfg, seed=seed, gamma_noise=gamma_noise)
    x = synth.activations(cfg, seed=seed)
    dy = synth.upstream_grad(cfg)
    dev = [{n: v.to(dtype).cuda() for n, v in W.items()} for W in host]
    return host, x, dy, dev, x.to(dtype).cuda(), dy.to(dtype).cuda()


def _compare(cfg, sched, step, fp32, granularity="per_sequence", gamma_noise=0.0, sublayer=False):
    dtype = torch.float32 if fp32 else torch.bfloat16
    host, x, dy, dev, xd, dyd = _inputs(cfg, dtype, gamma_noise)
    out, dX, grads, (mask, idx, cnt) = gpu_run(cfg, sched, step, dev, xd, dyd, granularity, fp32,
                                               sublayer=sublayer)
    rout, rdX, rgrads, rmask = oracle_run(cfg, sched, step, host, x, dy, granularity, sublayer=sublayer)
    assert (mask == rmask).all()
    ridx, rcnt = OM.kept_lists(rmask)
    assert (idx == ridx).all() and (cnt == rcnt).all()
    check_close("out", to_np(out), rout, fp32)
    check_close("dX", to_np(dX), rdX, fp32)
    for l in range(cfg["L"]):
        for n in grads[l]:
            check_close(f"layer{l}.{n}", to_np(grads[l][n]), rgrads[l][n], fp32)
    # dropped sequences: output and gradient pass through bit for bit
    for b in range(cfg["B"]):
        if not rmask[..., b].any():
            assert torch.equal(out.view(cfg["B"], cfg["S"], -1)[b].cpu(), xd.view(cfg["B"], cfg["S"], -1)[b].cpu())
            assert torch.equal(dX.view(cfg["B"], cfg["S"], -1)[b].cpu(), dyd.view(cfg["B"], cfg["S"], -1)[b].cpu())
    return mask


@pytest.mark.parametrize("fp32", [True, False], ids=["fp32", "bf16"])
def test_tiny_workload(fp32):
    cfg = synth.CONFIGS["tiny"]
    mask = _compare(cfg, synth.SCHEDULES["tiny"], 0, fp32)
    assert mask[0].all() and 0 < mask[1].sum() < cfg["B"]


@pytest.mark.parametrize("fp32", [True, False], ids=["fp32", "bf16"])
def test_tiny_gqa_gains_per_batch(fp32):
    cfg = dict(synth.CONFIGS["tiny"], H=4, Hkv=2, B=5, L=3)
    sched = dict(dist="uniform", p_max=0.5, time="const", seed=9)
    _compare(cfg, sched, 3, fp32, granularity="per_batch", gamma_noise=0.1)
    _compare(cfg, dict(sched, dist="ild"), 4, fp32, gamma_noise=0.1)


@pytest.mark.parametrize("fp32", [True, False], ids=["fp32", "bf16"])
def test_all_dropped_is_identity(fp32):
    cfg = synth.CONFIGS["tiny"]
    dtype = torch.float32 if fp32 else torch.bfloat16
    host, x, dy, dev, xd, dyd = _inputs(cfg, dtype)
    sched = dict(dist="uniform", p_max=1.0, time="const", seed=1)
    out, dX, grads, (mask, idx, cnt) = gpu_run(cfg, sched, 0, dev, xd, dyd, fp32_debug=fp32)
    assert not mask.any() and (cnt == 0).all() and (idx == -1).all()
    assert torch.equal(out, xd) and torch.equal(dX, dyd)
    for G in grads:
        for n, g in G.items():
            assert (g == 0).all(), n


@pytest.mark.parametrize("fp32", [True, False], ids=["fp32", "bf16"])
def test_ragged_kept_tiles(fp32):
    # S = 64 rows per sequence and odd kept counts: the last 128-row tile is
    # half empty; S = 192 makes tiles straddle sequences.
    for S, B in ((64, 7), (192, 3)):
        cfg = dict(synth.CONFIGS["tiny"], S=S, B=B, L=2, F=320, d=192, H=6, Hkv=3)
        sched = dict(dist="explicit", p_explicit=[0.3, 0.6], time="const", seed=5)
        _compare(cfg, sched, 1, fp32, gamma_noise=0.05)


MULTI = [
    dict(L=2, d=256, H=4, Hkv=2, Dh=64, F=512, B=3, S=512, eps=1e-6, rope_theta=1e4, alpha=1.0),
    dict(L=2, d=512, H=4, Hkv=1, Dh=128, F=768, B=2, S=1024, eps=1e-6, rope_theta=5e5, alpha=0.5),
]


@pytest.mark.parametrize("fp32", [True, False], ids=["fp32", "bf16"])
@pytest.mark.parametrize("cfg", MULTI, ids=["S512-dh64-gqa", "S1024-dh128-mqa"])
def test_multi_tile_full_tensors(cfg, fp32):
    # every attention and GEMM tile of several-tile sequences, compared on the
    # full tensors (not just the first rows)
    sched = dict(dist="explicit", p_explicit=[0.2, 0.5], time="const", seed=11)
    _compare(cfg, sched, 2, fp32, gamma_noise=0.1)


@pytest.mark.parametrize("fp32", [True, False], ids=["fp32", "bf16"])
def test_sublayer_granularity(fp32):
    # independent attention / FFN masks (Model Granularity subsection): every
    # combination of (attention kept, FFN kept) occurs; a block's gradients
    # sum over its own kept sequences
    cfg = dict(synth.CONFIGS["tiny"], L=3, B=8, H=4, Hkv=2)
    sched = dict(dist="uniform", p_max=0.5, time="const", seed=3)
    mask = _compare(cfg, sched, 5, fp32, gamma_noise=0.1, sublayer=True)
    assert mask.shape == (2, 3, 8)
    combos = {(int(a), int(f)) for a, f in zip(mask[0].ravel(), mask[1].ravel())}
    assert combos == {(0, 0), (0, 1), (1, 0), (1, 1)}


@pytest.mark.parametrize("fp32", [True, False], ids=["fp32", "bf16"])
def test_sublayer_multi_tile(fp32):
    cfg = MULTI[1]
    sched = dict(dist="explicit", p_explicit=[0.5, 0.5], time="const", seed=21)
    _compare(cfg, sched, 0, fp32, gamma_noise=0.1, sublayer=True, granularity="per_sequence")


PAPER = [
    # ALiBi + squared ReLU; tiny shape (mma.sync attention, Dh 32)
    dict(synth.CONFIGS["tiny"], H=4, Hkv=2, rope_theta=0.0, alibi=True, act="relu2"),
    # 6 heads (slopes of a non-power-of-two head count), tcgen05 forward, mma.sync backward
    dict(L=2, d=384, H=6, Hkv=3, Dh=64, F=1536, B=3, S=512, eps=1e-6, rope_theta=0.0, alpha=1.0, alibi=True,
         act="relu2"),
    # tcgen05 forward and backward
    dict(L=2, d=512, H=4, Hkv=1, Dh=128, F=1024, B=2, S=1024, eps=1e-6, rope_theta=0.0, alpha=1.0, alibi=True,
         act="relu2"),
]


@pytest.mark.parametrize("fp32", [True, False], ids=["fp32", "bf16"])
@pytest.mark.parametrize("cfg", PAPER, ids=["tiny", "S512-dh64-h6", "S1024-dh128"])
def test_paper_architecture(cfg, fp32):
    sched = dict(dist="explicit", p_explicit=[0.3, 0.5][: cfg["L"]], time="const", seed=13)
    _compare(cfg, sched, 1, fp32, gamma_noise=0.1)


@pytest.mark.parametrize("fp32", [True, False], ids=["fp32", "bf16"])
def test_paper_architecture_sublayer(fp32):
    cfg = PAPER[2]
    sched = dict(dist="explicit", p_explicit=[0.5, 0.5], time="const", seed=21)
    _compare(cfg, sched, 0, fp32, gamma_noise=0.1, sublayer=True)
