"""Pins of the oracle's per-token granularity (masks [L, B, S]; the Tensor
Granularity subsection leaves per-token dropping to future work, and
oracle/masks.py states the reading) against things fixed independently of it:
  * a torch composition of dense layers (library rms_norm, SDPA, complex
    RoPE at the kept tokens' positions) differentiated by autograd;
  * reductions: all tokens kept is the dense stack; a mask constant along
    each sequence is the per-sequence stack;
  * relative positions: a kept contiguous block equals the dense layer run on
    that block alone (rotary embedding and ALiBi depend on distances only);
  * a dropped token neither changes nor feeds any kept token at that layer;
  * central finite differences of the per-token stack in float64;
  * the draw: Philox words 2 / 3 at the global token index, exact threshold
    edges, b_offset shifting the token index, the kept fraction."""

import numpy as np
import pytest
import torch

from oracle import masks as M
from oracle import stack as O
from torch_reference import to_torch_layers, token_masked_stack

MICRO = dict(L=2, d=32, H=4, Hkv=2, Dh=8, F=48, B=3, S=12, eps=1e-6, rope_theta=1e4, alpha=1.0)
PAPER_ARCH = dict(MICRO, alibi=True, rope_theta=0.0, act="relu2")


def _layers(cfg, seed=0):
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(cfg["L"]):
        W = {}
        for n in O.WEIGHT_NAMES:
            shp = O.shape_of(cfg, n)
            W[n] = 1.0 + 0.1 * rng.standard_normal(shp) if n in ("g1", "g2") else 0.2 * rng.standard_normal(shp)
        out.append(W)
    return out


def _inputs(cfg, seed=1):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((cfg["B"], cfg["S"], cfg["d"])), rng.standard_normal((cfg["B"], cfg["S"], cfg["d"]))


def _random_masks(cfg, seed, p=0.4, sublayer=False):
    rng = np.random.default_rng(seed)
    shape = ((2,) if sublayer else ()) + (cfg["L"], cfg["B"], cfg["S"])
    return (rng.random(shape) >= p).astype(np.uint8)


def _slopes(cfg):
    return O.alibi_slopes(cfg["H"]) if cfg.get("alibi") else None


def _run(cfg, layers, x, dy, masks, scales):
    out, caches = O.stack_forward(x, layers, cfg, masks, scales, per_token=True)
    dX, grads = O.stack_backward(dy, layers, cfg, masks, scales, caches, per_token=True)
    return out, dX, grads


@pytest.mark.parametrize("cfg,sublayer", [(MICRO, False), (MICRO, True), (PAPER_ARCH, False)],
                         ids=["rope-swiglu", "rope-swiglu-sublayer", "alibi-relu2"])
def test_per_token_matches_torch_autograd(cfg, sublayer):
    layers = _layers(cfg, seed=3)
    x, dy = _inputs(cfg, seed=4)
    masks = _random_masks(cfg, seed=5, sublayer=sublayer)
    scales = [1.0 / (1 - 0.4), 1.3]
    out, dX, grads = _run(cfg, layers, x, dy, masks, scales)
    tl = to_torch_layers(layers, requires_grad=True)
    tx = torch.tensor(x, requires_grad=True)
    tout = token_masked_stack(tx, tl, cfg, masks, scales, _slopes(cfg))
    np.testing.assert_allclose(out, tout.detach().numpy(), rtol=0, atol=1e-11)
    (tout * torch.tensor(dy)).sum().backward()
    np.testing.assert_allclose(dX, tx.grad.numpy(), rtol=0, atol=1e-10)
    for l in range(cfg["L"]):
        for n in O.WEIGHT_NAMES:
            ref = tl[l][n].grad
            ref = np.zeros(O.shape_of(cfg, n)) if ref is None else ref.numpy()
            np.testing.assert_allclose(grads[l][n], ref, rtol=0, atol=1e-10, err_msg=f"layer {l} {n}")


def test_reductions_to_dense_and_per_sequence():
    cfg = MICRO
    layers = _layers(cfg, seed=6)
    x, dy = _inputs(cfg, seed=7)
    scales = [1.25, 2.0]
    # every token kept == every sequence kept
    ones = np.ones((cfg["L"], cfg["B"], cfg["S"]), dtype=np.uint8)
    o1, d1, g1 = _run(cfg, layers, x, dy, ones, scales)
    c = O.stack_forward(x, layers, cfg, np.ones((cfg["L"], cfg["B"]), dtype=np.uint8), scales)
    o2 = c[0]
    d2, g2 = O.stack_backward(dy, layers, cfg, np.ones((cfg["L"], cfg["B"]), dtype=np.uint8), scales, c[1])
    np.testing.assert_allclose(o1, o2, rtol=0, atol=1e-12)
    np.testing.assert_allclose(d1, d2, rtol=0, atol=1e-12)
    # a mask constant along each sequence == the per-sequence stack
    seq = np.array([[1, 0, 1], [0, 1, 1]], dtype=np.uint8)
    tok = np.repeat(seq[:, :, None], cfg["S"], axis=2)
    o1, d1, g1 = _run(cfg, layers, x, dy, tok, scales)
    c = O.stack_forward(x, layers, cfg, seq, scales)
    d2, g2 = O.stack_backward(dy, layers, cfg, seq, scales, c[1])
    np.testing.assert_allclose(o1, c[0], rtol=0, atol=1e-12)
    np.testing.assert_allclose(d1, d2, rtol=0, atol=1e-12)
    for l in range(cfg["L"]):
        for n in O.WEIGHT_NAMES:
            np.testing.assert_allclose(g1[l][n], g2[l][n], rtol=0, atol=1e-12)


@pytest.mark.parametrize("cfg", [MICRO, PAPER_ARCH], ids=["rope", "alibi"])
def test_contiguous_block_is_position_free(cfg):
    # Keeping tokens s0 .. s0+n-1 of one sequence equals running the dense
    # layer on that block as its own sequence at positions 0 .. n-1: the
    # rotary embedding and the ALiBi bias see distances only.
    cfg = dict(cfg, L=1, B=1)
    layers = _layers(cfg, seed=8)
    x, dy = _inputs(cfg, seed=9)
    s0, n = 5, 6
    mask = np.zeros((1, 1, cfg["S"]), dtype=np.uint8)
    mask[0, 0, s0 : s0 + n] = 1
    out, dX, grads = _run(cfg, layers, x, dy, mask, [1.5])
    sub = dict(cfg, S=n)
    c = O.stack_forward(x[:, s0 : s0 + n], layers, sub, np.ones((1, 1), dtype=np.uint8), [1.5])
    d2, g2 = O.stack_backward(dy[:, s0 : s0 + n], layers, sub, np.ones((1, 1), dtype=np.uint8), [1.5], c[1])
    np.testing.assert_allclose(out[:, s0 : s0 + n], c[0], rtol=0, atol=1e-11)
    np.testing.assert_allclose(dX[:, s0 : s0 + n], d2, rtol=0, atol=1e-11)
    for n_ in O.WEIGHT_NAMES:
        np.testing.assert_allclose(grads[0][n_], g2[0][n_], rtol=0, atol=1e-11)
    outside = np.ones(cfg["S"], dtype=bool)
    outside[s0 : s0 + n] = False
    assert (out[0, outside] == x[0, outside]).all() and (dX[0, outside] == dy[0, outside]).all()


def test_dropped_token_is_invisible():
    # At L = 1 a dropped token keeps its input and changing it changes no
    # kept token's output (it contributes no key or value).
    cfg = dict(MICRO, L=1)
    layers = _layers(cfg, seed=10)
    x, _ = _inputs(cfg, seed=11)
    mask = _random_masks(cfg, seed=12, p=0.5)
    b, s = np.argwhere(mask[0] == 0)[0]
    out1, _ = O.stack_forward(x, layers, cfg, mask, [1.7], per_token=True)
    x2 = x.copy()
    x2[b, s] += 3.0
    out2, _ = O.stack_forward(x2, layers, cfg, mask, [1.7], per_token=True)
    kept = mask[0] == 1
    np.testing.assert_array_equal(out1[kept], out2[kept])
    assert (out2[b, s] == x2[b, s]).all() and (out1[~kept] == x[~kept]).all()


def test_finite_differences_per_token():
    cfg = dict(MICRO, B=2, S=8)
    layers = _layers(cfg, seed=13)
    x, dy = _inputs(cfg, seed=14)
    masks = _random_masks(cfg, seed=15, p=0.35, sublayer=True)
    scales = [1.3, 0.8]
    out, dX, grads = _run(cfg, layers, x, dy, masks, scales)
    rng = np.random.default_rng(16)
    eps = 1e-5

    def f(xx, lay):
        return float(np.sum(O.stack_forward(xx, lay, cfg, masks, scales, per_token=True)[0] * dy))

    v = rng.standard_normal(x.shape)
    num = (f(x + eps * v, layers) - f(x - eps * v, layers)) / (2 * eps)
    assert abs(num - np.sum(dX * v)) <= 1e-7 * max(1.0, abs(num))
    for l, n in ((0, "w_qkv"), (1, "w_gu"), (0, "g1"), (1, "w_o")):
        vw = rng.standard_normal(O.shape_of(cfg, n))
        lp = [dict(W) for W in layers]
        lm = [dict(W) for W in layers]
        lp[l][n] = layers[l][n] + eps * vw
        lm[l][n] = layers[l][n] - eps * vw
        num = (f(x, lp) - f(x, lm)) / (2 * eps)
        assert abs(num - np.sum(grads[l][n] * vw)) <= 1e-7 * max(1.0, abs(num)), (l, n)


def test_token_draw_words_and_edges():
    seed, step, S = 2024, 9, 5
    thr = [int(0.3 * 2**32), int(0.6 * 2**32)]
    m = M.draw_masks(seed, step, thr, 4, M.PER_TOKEN, S=S)
    assert m.shape == (2, 4, S) and m.dtype == np.uint8
    for l in range(2):
        for b in range(4):
            for s in range(S):
                u = M.token_word(seed, step, l, b * S + s)
                assert m[l, b, s] == (1 if u >= thr[l] else 0)
    # the word at the global token index is word 2 of the Philox output
    assert M.token_word(seed, step, 1, 17) == M.mask_word(seed, step, 1, 17, 2)
    # exact threshold edges (keep iff u >= thr)
    u = M.token_word(seed, step, 0, 3)
    assert M.draw_masks(seed, step, [u], 1, M.PER_TOKEN, S=S)[0, 0, 3] == 1
    assert M.draw_masks(seed, step, [u + 1], 1, M.PER_TOKEN, S=S)[0, 0, 3] == 0
    # a shard's tokens are the global tokens shifted by b_offset * S
    full = M.draw_masks(seed, step, thr, 6, M.PER_TOKEN, S=S)
    shard = M.draw_masks(seed, step, thr, 2, M.PER_TOKEN, b_offset=3, S=S)
    assert (shard == full[:, 3:5]).all()
    # sub-layer: attention mask = the layer mask (word 2), FFN mask from word 3
    pair = M.draw_masks(seed, step, thr, 4, M.PER_TOKEN, sublayer=True, S=S)
    assert (pair[0] == m).all()
    assert pair[1, 1, 2, 4] == (1 if M.mask_word(seed, step, 1, 2 * S + 4, 3) >= thr[1] else 0)


def test_token_draw_rate_and_lists():
    p = 0.3
    m = M.draw_masks(77, 3, [int(p * 2**32)], 64, M.PER_TOKEN, S=2048)
    n = m.size
    kept = int(m.sum())
    sigma = np.sqrt(n * p * (1 - p))
    assert abs(kept - n * (1 - p)) <= 5 * sigma
    small = M.draw_masks(5, 1, [int(0.5 * 2**32)] * 2, 3, M.PER_TOKEN, S=7)
    rows, cnt, seg = M.kept_token_lists(small)
    for l in range(2):
        ref = [b * 7 + s for b in range(3) for s in range(7) if small[l, b, s]]
        assert cnt[l] == len(ref) and list(rows[l, : cnt[l]]) == ref and (rows[l, cnt[l]:] == -1).all()
        assert seg[l, 0] == 0 and seg[l, -1] == cnt[l]
        assert list(np.diff(seg[l])) == [int(small[l, b].sum()) for b in range(3)]
