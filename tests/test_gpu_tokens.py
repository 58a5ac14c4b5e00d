"""Per-token granularity through the C ABI against the oracle: the masks and
kept-token lists bit for bit (Philox words 2 / 3 at the global token index,
sub-layer tables, shard offsets), and the whole stack forward and backward on
the float32 debug path (SIMT attention, tolerance 1e-5 of each tensor's max)
and the bf16 path (tcgen05 attention with ragged per-sequence segments,
2e-2 of max + 1e-3), plus the exact cases: every token kept equals the
per-sequence stack, every token dropped is the identity."""

import numpy as np
import pytest
import torch

import paper_2609_05275_gb300 as P
from paper_2609_05275_gb300 import synth
from parity import check_close, gpu_run, oracle_masks, oracle_run, to_np
from oracle import masks as OM

pytestmark = pytest.mark.gpu

# Dh = 128 and S % 128 == 0: the bf16 path's tcgen05 attention; S = 384 with
# p ~ 0.5 gives segments of every length mod 128
TOK = dict(L=2, d=256, H=2, Hkv=1, Dh=128, F=512, B=3, S=384, eps=1e-6, rope_theta=1e4, alpha=1.0)
# head size 64: the tcgen05 forward and the two-kernel backward at Dh = 64
TOK64 = dict(TOK, H=4, Hkv=2, Dh=64)
TINY = synth.CONFIGS["tiny"]


def _inputs(cfg, dtype, seed=0):
    host = synth.stack_weights(cfg, seed=seed, gamma_noise=0.1)
    x = synth.activations(cfg, seed=seed)
    dy = synth.upstream_grad(cfg)
    dev = [{n: v.to(dtype).cuda() for n, v in W.items()} for W in host]
    return host, x, dy, dev, x.to(dtype).cuda(), dy.to(dtype).cuda()


def _check_lists(mask, idx, cnt, rmask):
    assert mask.shape == rmask.shape and (mask == rmask).all()
    rrows, rcnt, _ = OM.kept_token_lists(rmask)
    assert (cnt == rcnt).all()
    assert (idx == rrows).all()


@pytest.mark.parametrize("sublayer", [False, True], ids=["layer", "sublayer"])
def test_token_masks_bit_exact(sublayer):
    cfg = dict(TINY, L=4, B=5)
    sched = dict(dist="ild", p_max=0.7, time="its", T=100, seed=12345)
    st = P.LayerDropStack(cfg, sched, granularity="per_token", fp32_debug=True, sublayer=sublayer)
    try:
        for t in (0, 1, 57, 99):
            mask, idx, cnt = st.draw_masks(t)
            rmask, _, _ = oracle_masks(cfg, sched, t, "per_token", sublayer)
            _check_lists(mask, idx, cnt, rmask)
    finally:
        st.close()


def test_token_masks_shard_offset():
    cfg = dict(TINY, L=3, B=2)
    sched = dict(dist="uniform", p_max=0.5, time="const", seed=77)
    st = P.LayerDropStack(cfg, sched, granularity="per_token", fp32_debug=True, b_offset=5)
    try:
        mask, idx, cnt = st.draw_masks(3)
        rates = [0.5] * 3
        thr = [int(np.floor(p * 2**32)) for p in rates]
        ref = OM.draw_masks(77, 3, thr, 2, OM.PER_TOKEN, b_offset=5, S=cfg["S"])
        _check_lists(mask, idx, cnt, ref)
    finally:
        st.close()


def _compare(cfg, sched, step, fp32, sublayer=False):
    dtype = torch.float32 if fp32 else torch.bfloat16
    host, x, dy, dev, xd, dyd = _inputs(cfg, dtype)
    out, dX, grads, (mask, idx, cnt) = gpu_run(cfg, sched, step, dev, xd, dyd, "per_token", fp32, sublayer=sublayer)
    rout, rdX, rgrads, rmask = oracle_run(cfg, sched, step, host, x, dy, "per_token", sublayer=sublayer)
    _check_lists(mask, idx, cnt, rmask)
    check_close("out", to_np(out), rout, fp32)
    check_close("dX", to_np(dX), rdX, fp32)
    for l in range(cfg["L"]):
        for n in grads[l]:
            check_close(f"layer{l}.{n}", to_np(grads[l][n]), rgrads[l][n], fp32)
    # tokens dropped at every layer: output and gradient bit for bit
    dropped = ~(rmask.reshape(-1, cfg["B"] * cfg["S"]).any(axis=0))
    o2, x2 = out.view(cfg["B"] * cfg["S"], -1).cpu(), xd.view(cfg["B"] * cfg["S"], -1).cpu()
    d2, y2 = dX.view(cfg["B"] * cfg["S"], -1).cpu(), dyd.view(cfg["B"] * cfg["S"], -1).cpu()
    for r in np.nonzero(dropped)[0]:
        assert torch.equal(o2[r], x2[r]) and torch.equal(d2[r], y2[r])
    return rmask


@pytest.mark.parametrize("sublayer", [False, True], ids=["layer", "sublayer"])
def test_token_stack_fp32(sublayer):
    sched = dict(dist="explicit", p_max=0.0, p_explicit=[0.3, 0.6], time="const", seed=3)
    _compare(TINY, sched, 1, True, sublayer)


@pytest.mark.parametrize("dh", [128, 64], ids=["dh128", "dh64"])
@pytest.mark.parametrize("sublayer", [False, True], ids=["layer", "sublayer"])
def test_token_stack_bf16(sublayer, dh):
    cfg = TOK if dh == 128 else TOK64
    sched = dict(dist="explicit", p_max=0.0, p_explicit=[0.45, 0.55], time="const", seed=5)
    rmask = _compare(cfg, sched, 2, False, sublayer)
    lens = rmask.reshape(-1, cfg["B"], cfg["S"]).sum(axis=2)
    assert (lens % 128 != 0).any()  # ragged segments: tiles straddle sequence ends


def test_token_stack_bf16_fp32_agree_on_gqa():
    # grouped-query heads (H = 4, Hkv = 2) and a third layer
    cfg = dict(TOK, H=4, Hkv=2, L=3, B=2)
    sched = dict(dist="uniform", p_max=0.35, time="const", seed=8)
    _compare(cfg, sched, 0, False)


@pytest.mark.parametrize("fp32,dh", [(True, 32), (False, 128), (False, 64)], ids=["fp32", "bf16", "bf16-dh64"])
def test_token_all_kept_equals_per_sequence(fp32, dh):
    cfg = TINY if fp32 else (TOK if dh == 128 else TOK64)
    dtype = torch.float32 if fp32 else torch.bfloat16
    host, x, dy, dev, xd, dyd = _inputs(cfg, dtype)
    sched = dict(dist="uniform", p_max=0.0, time="const", seed=1)
    a = gpu_run(cfg, sched, 0, dev, xd, dyd, "per_token", fp32)
    b = gpu_run(cfg, sched, 0, dev, xd, dyd, "per_sequence", fp32)
    assert a[3][0].all() and (a[3][2] == cfg["B"] * cfg["S"]).all()
    assert torch.equal(a[0], b[0])
    assert (a[1].float() - b[1].float()).abs().max().item() <= 1e-2 * b[1].float().abs().max().item() + 1e-6
    for Ga, Gb in zip(a[2], b[2]):
        for n in Ga:
            assert (Ga[n] - Gb[n]).abs().max().item() <= 1e-2 * Gb[n].abs().max().item() + 1e-6, n


@pytest.mark.parametrize("fp32", [True, False], ids=["fp32", "bf16"])
def test_token_all_dropped_is_identity(fp32):
    cfg = TINY if fp32 else TOK
    dtype = torch.float32 if fp32 else torch.bfloat16
    host, x, dy, dev, xd, dyd = _inputs(cfg, dtype)
    sched = dict(dist="uniform", p_max=1.0, time="const", seed=1)
    out, dX, grads, (mask, idx, cnt) = gpu_run(cfg, sched, 0, dev, xd, dyd, "per_token", fp32)
    assert not mask.any() and (cnt == 0).all() and (idx == -1).all()
    assert torch.equal(out, xd) and torch.equal(dX, dyd)
    for G in grads:
        for n, g in G.items():
            assert (g == 0).all(), n


@pytest.mark.parametrize("fp32,dh", [(True, 32), (False, 128), (False, 64)], ids=["fp32", "bf16", "bf16-dh64"])
def test_token_tiny_and_empty_segments(fp32, dh):
    # p close to 1 over short sequences: segments of 0, 1, 2, ... kept tokens
    # side by side (a sequence with none, its neighbours with a few)
    cfg = dict(TINY, B=16, S=64) if fp32 else dict(TOK if dh == 128 else TOK64, B=16, S=128, L=2)
    sched = dict(dist="uniform", p_max=0.985 if not fp32 else 0.97, time="const", seed=21)
    rmask = _compare(cfg, sched, 0, fp32)
    lens = rmask.reshape(-1, cfg["B"], cfg["S"]).sum(axis=2)
    assert (lens == 0).any() and (lens > 0).any() and (lens <= 3).any()
