"""Pins of the oracle's decoder stack (forward and hand-derived backward)
against things fixed independently of it:
  * a dense decoder written with torch library routines (rms_norm, SDPA,
    complex RoPE, silu) and differentiated by autograd;
  * brute force over every mask of a 2-sequence, 2-layer stack, composed
    from that dense layer per the case form of the Preliminary section;
  * central finite differences in float64;
  * p = 1 gives the identity (dX = dY, dW = 0) exactly;
  * causality and sequence independence, the two properties the full-size
    parity protocol relies on."""

import itertools
import os

import numpy as np
import pytest
import torch

from oracle import stack as O
from torch_reference import masked_stack, to_torch_layers

MICRO = dict(L=2, d=32, H=4, Hkv=2, Dh=8, F=48, B=3, S=8, eps=1e-6, rope_theta=1e4, alpha=1.0)


def _layers(cfg, seed=0, gamma_noise=0.1):
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(cfg["L"]):
        W = {}
        for n in O.WEIGHT_NAMES:
            shp = O.shape_of(cfg, n)
            if n in ("g1", "g2"):
                W[n] = 1.0 + gamma_noise * rng.standard_normal(shp)
            else:
                W[n] = 0.2 * rng.standard_normal(shp)
        out.append(W)
    return out


def _inputs(cfg, seed=1):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((cfg["B"], cfg["S"], cfg["d"]))
    dy = rng.standard_normal((cfg["B"], cfg["S"], cfg["d"]))
    return x, dy


PAPER_ARCH = dict(MICRO, alibi=True, rope_theta=0.0, act="relu2")  # ALiBi + squared ReLU (Methodology)

CFGS = [
    MICRO,
    dict(MICRO, H=4, Hkv=4, rope_theta=0.0),   # MHA, no rotary embedding
    dict(MICRO, H=4, Hkv=1, Dh=16, d=48),      # one key/value head
    PAPER_ARCH,                                # ALiBi + squared ReLU, 4 heads
    dict(PAPER_ARCH, H=6, Hkv=3),              # ALiBi slopes for a head count that is not a power of two
]


def _slopes(cfg):
    return O.alibi_slopes(cfg["H"]) if cfg.get("alibi") else None


@pytest.mark.parametrize("cfg", CFGS, ids=["gqa-rope", "mha-norope", "mqa", "alibi-relu2", "alibi6-relu2"])
def test_forward_and_backward_match_torch_autograd(cfg):
    layers = _layers(cfg)
    x, dy = _inputs(cfg)
    masks = np.array([[1, 0, 1], [1, 1, 0]], dtype=np.uint8)
    scales = [1.0 / (1 - 0.3), 1.7]
    out, caches = O.stack_forward(x, layers, cfg, masks, scales)
    dX, grads = O.stack_backward(dy, layers, cfg, masks, scales, caches)

    tl = to_torch_layers(layers, requires_grad=True)
    tx = torch.tensor(x, requires_grad=True)
    tout = masked_stack(tx, tl, cfg, masks, scales, _slopes(cfg))
    np.testing.assert_allclose(out, tout.detach().numpy(), rtol=0, atol=1e-11)
    (tout * torch.tensor(dy)).sum().backward()
    np.testing.assert_allclose(dX, tx.grad.numpy(), rtol=0, atol=1e-10)
    for l in range(cfg["L"]):
        for n in O.WEIGHT_NAMES:
            np.testing.assert_allclose(grads[l][n], tl[l][n].grad.numpy(), rtol=0, atol=1e-10,
                                       err_msg=f"layer {l} {n}")


def test_all_masks_brute_force():
    # Every mask of B = 2, L = 2 (16 cases) against the per-sequence case form.
    cfg = dict(MICRO, B=2)
    layers = _layers(cfg, seed=3)
    x, _ = _inputs(cfg, seed=4)
    tl = to_torch_layers(layers)
    scales = [1.25, 2.0]
    for bits in itertools.product([0, 1], repeat=4):
        masks = np.array(bits, dtype=np.uint8).reshape(2, 2)
        out, _ = O.stack_forward(x, layers, cfg, masks, scales)
        ref = masked_stack(torch.tensor(x), tl, cfg, masks, scales).numpy()
        np.testing.assert_allclose(out, ref, rtol=0, atol=1e-11)
        for b in range(2):
            if not masks[:, b].any():
                assert (out[b] == x[b]).all()


def test_sublayer_matches_torch_autograd():
    # Independent attention / FFN masks (every combination occurs): forward
    # and hand-derived backward against the dense composition + autograd.
    cfg = MICRO
    layers = _layers(cfg, seed=8)
    x, dy = _inputs(cfg, seed=9)
    masks = np.array([[[1, 0, 1], [0, 1, 1]],     # M_attn [L, B]
                      [[0, 0, 1], [1, 1, 0]]],    # M_ffn
                     dtype=np.uint8)
    scales = [1.0 / (1 - 0.4), 1.3]
    out, caches = O.stack_forward(x, layers, cfg, masks, scales)
    dX, grads = O.stack_backward(dy, layers, cfg, masks, scales, caches)
    tl = to_torch_layers(layers, requires_grad=True)
    tx = torch.tensor(x, requires_grad=True)
    tout = masked_stack(tx, tl, cfg, masks, scales)
    np.testing.assert_allclose(out, tout.detach().numpy(), rtol=0, atol=1e-11)
    (tout * torch.tensor(dy)).sum().backward()
    np.testing.assert_allclose(dX, tx.grad.numpy(), rtol=0, atol=1e-10)
    for l in range(cfg["L"]):
        for n in O.WEIGHT_NAMES:
            ref = tl[l][n].grad
            ref = np.zeros(O.shape_of(cfg, n)) if ref is None else ref.numpy()
            np.testing.assert_allclose(grads[l][n], ref, rtol=0, atol=1e-10, err_msg=f"layer {l} {n}")


def test_sublayer_brute_force_and_layer_reduction():
    # Every (M_attn, M_ffn) of B = 1, L = 2 (16 cases) against the dense
    # composition; equal masks reproduce the layer-granularity stack exactly.
    cfg = dict(MICRO, B=1)
    layers = _layers(cfg, seed=10)
    x, dy = _inputs(cfg, seed=11)
    tl = to_torch_layers(layers)
    scales = [1.25, 2.0]
    for bits in itertools.product([0, 1], repeat=4):
        masks = np.array(bits, dtype=np.uint8).reshape(2, 2, 1)
        out, _ = O.stack_forward(x, layers, cfg, masks, scales)
        ref = masked_stack(torch.tensor(x), tl, cfg, masks, scales).numpy()
        np.testing.assert_allclose(out, ref, rtol=0, atol=1e-11)
    for bits in itertools.product([0, 1], repeat=2):
        m = np.array(bits, dtype=np.uint8).reshape(2, 1)
        o1, c1 = O.stack_forward(x, layers, cfg, m, scales)
        o2, c2 = O.stack_forward(x, layers, cfg, np.stack([m, m]), scales)
        d1, g1 = O.stack_backward(dy, layers, cfg, m, scales, c1)
        d2, g2 = O.stack_backward(dy, layers, cfg, np.stack([m, m]), scales, c2)
        assert (o1 == o2).all() and (d1 == d2).all()
        assert all((g1[l][n] == g2[l][n]).all() for l in range(2) for n in O.WEIGHT_NAMES)


@pytest.mark.parametrize("cfg", [MICRO, PAPER_ARCH], ids=["rope-swiglu", "alibi-relu2"])
def test_eval_forward_early_exit_and_skipping(cfg):
    # Eq. (transformer_layer_dropout_eval) against the dense torch
    # composition: early exit at l' = the first l' layers at scale r_eval;
    # intermediate skipping = those layers with the others left out.
    cfg = dict(cfg, L=4)
    layers = _layers(cfg, seed=12)
    x, _ = _inputs(cfg, seed=13)
    tl = to_torch_layers(layers)
    tx = torch.tensor(x)
    B = cfg["B"]
    for execute, r_eval in (([1, 1, 1, 1], None), ([1, 1, 0, 0], None), ([1, 0, 1, 0], [1.0, 9.0, 0.5, 9.0]),
                            ([0, 1, 1, 1], [1.0, 0.7, 1.3, 2.0])):
        out = O.stack_forward_eval(x, layers, cfg, execute, r_eval)
        masks = np.repeat(np.array(execute, dtype=np.uint8)[:, None], B, axis=1)
        scales = [1.0] * 4 if r_eval is None else r_eval
        ref = masked_stack(tx, tl, cfg, masks, scales, _slopes(cfg)).numpy()
        np.testing.assert_allclose(out, ref, rtol=0, atol=1e-11)
    assert (O.stack_forward_eval(x, layers, cfg, [0, 0, 0, 0]) == x).all()


def test_p1_is_identity():
    cfg = MICRO
    layers = _layers(cfg)
    x, dy = _inputs(cfg)
    masks = np.zeros((cfg["L"], cfg["B"]), dtype=np.uint8)
    out, caches = O.stack_forward(x, layers, cfg, masks, [0.0, 0.0])
    dX, grads = O.stack_backward(dy, layers, cfg, masks, [0.0, 0.0], caches)
    assert (out == x).all() and (dX == dy).all()
    assert all((g[n] == 0).all() for g in grads for n in O.WEIGHT_NAMES)


def test_alibi_slopes():
    # ALiBi paper (Press et al., ICLR 2022), Section 3: 8 heads use 2^-1 ..
    # 2^-8; 16 heads the sequence that starts at 2^-0.5 with ratio 2^-0.5
    # (tests/golden/alibi_slopes.txt).  Other head counts: the slopes of the
    # largest power of two n0 <= H, then geometric means of neighbouring
    # slopes of that sequence (1 taken as the slope before the first).
    gold = {}
    for line in open(os.path.join(os.path.dirname(__file__), "golden", "alibi_slopes.txt")):
        if line.strip() and not line.startswith("#"):
            h, *v = line.split()
            gold[int(h)] = [float(x) for x in v]
    for H, ref in gold.items():
        np.testing.assert_array_equal(O.alibi_slopes(H), np.array(ref))
    for H in (3, 5, 6, 9, 10, 12, 14, 21, 24, 40):
        m = O.alibi_slopes(H)
        n0 = 2 ** int(np.floor(np.log2(H)))
        base = O.alibi_slopes(n0)
        np.testing.assert_array_equal(m[:n0], base)
        prev = np.concatenate([[1.0], base])
        np.testing.assert_allclose(m[n0:], np.sqrt(prev[:-1] * prev[1:])[: H - n0], rtol=1e-15)
        assert len(set(m)) == H and (m > 0).all() and (m < 1).all()


def test_finite_differences_paper_arch():
    _finite_differences(dict(PAPER_ARCH, H=6, Hkv=2))


def test_finite_differences():
    _finite_differences(MICRO)


def _finite_differences(cfg):
    layers = _layers(cfg, seed=5)
    x, dy = _inputs(cfg, seed=6)
    masks = np.array([[1, 1, 0], [0, 1, 1]], dtype=np.uint8)
    scales = [1.5, 1.25]

    def loss(xx, ll):
        out, _ = O.stack_forward(xx, ll, cfg, masks, scales)
        return float((out * dy).sum())

    out, caches = O.stack_forward(x, layers, cfg, masks, scales)
    dX, grads = O.stack_backward(dy, layers, cfg, masks, scales, caches)
    rng = np.random.default_rng(7)
    h = 1e-6
    for _ in range(12):
        i = tuple(int(rng.integers(0, n)) for n in x.shape)
        xp, xm = x.copy(), x.copy()
        xp[i] += h
        xm[i] -= h
        fd = (loss(xp, layers) - loss(xm, layers)) / (2 * h)
        assert fd == pytest.approx(dX[i], rel=1e-5, abs=1e-6)
    for l in range(cfg["L"]):
        for n in O.WEIGHT_NAMES:
            for _ in range(3):
                shp = O.shape_of(cfg, n)
                i = tuple(int(rng.integers(0, s)) for s in shp)
                lp = [dict(W) for W in layers]
                lm = [dict(W) for W in layers]
                lp[l][n] = layers[l][n].copy()
                lm[l][n] = layers[l][n].copy()
                lp[l][n][i] += h
                lm[l][n][i] -= h
                fd = (loss(x, lp) - loss(x, lm)) / (2 * h)
                assert fd == pytest.approx(grads[l][n][i], rel=1e-5, abs=1e-6), (l, n, i)


def test_causal_truncation_and_independence():
    # Output rows < R depend only on input rows < R of the same sequence, and
    # with dY zero beyond row R the gradients come from rows < R only.
    cfg = dict(MICRO, S=16)
    layers = _layers(cfg, seed=8)
    x, dy = _inputs(cfg, seed=9)
    R = 5
    dy[:, R:, :] = 0.0
    masks = np.array([[1, 0, 1], [1, 1, 1]], dtype=np.uint8)
    scales = [1.2, 1.0]
    out, caches = O.stack_forward(x, layers, cfg, masks, scales)
    dX, grads = O.stack_backward(dy, layers, cfg, masks, scales, caches)
    tout, tcaches = O.stack_forward(x[:, :R], layers, cfg, masks, scales)
    tdX, tgrads = O.stack_backward(dy[:, :R], layers, cfg, masks, scales, tcaches)
    np.testing.assert_allclose(out[:, :R], tout, rtol=0, atol=1e-12)
    np.testing.assert_allclose(dX[:, :R], tdX, rtol=0, atol=1e-12)
    assert (dX[:, R:] == 0).all()
    for l in range(cfg["L"]):
        for n in O.WEIGHT_NAMES:
            np.testing.assert_allclose(grads[l][n], tgrads[l][n], rtol=0, atol=1e-11)
    # sequence independence
    x2 = x.copy()
    x2[1] += 1.0
    out2, _ = O.stack_forward(x2, layers, cfg, masks, scales)
    assert (out2[0] == out[0]).all() and (out2[2] == out[2]).all()
    assert not np.allclose(out2[1], out[1])
