"""Forward and backward of a pre-norm decoder stack under layer dropout.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

Follows Eq. (transformer_layer_dropout_train) with one mask per layer for
both sub-blocks (layer granularity, Model Granularity subsection):

    Z^l      = X^l + r M^l f_attn(X^l)
    X^{l+1}  = Z^l + r M^l f_ffn(Z^l)

or, with sub-layer granularity (same subsection), independent masks
M^l_attn and M^l_ffn in place of M^l in the two lines: a sequence may run
either block alone, both or neither.

and the per-sequence case form of the Preliminary section: a dropped
sequence keeps X^{l+1}[b] = X^l[b]; a kept one gets the residual update with
r = alpha / (1 - p^{l,t}) (Dropout Scale paragraph and the parameterization
table's residual rows).  Only kept sequences are evaluated, as in the
"efficient implementation" paragraph.

The paper leaves the block internals open (its footnote to the transformer
form); the block here is the one the workloads name: RMSNorm (eps inside the
square root, gain gamma), rotary position embedding on q and k, causal
grouped-query attention with scale 1/sqrt(Dh), SwiGLU feed-forward
h = silu(g) * u, no biases.  The paper's own models (Methodology section)
use ALiBi position biases and squared-ReLU activations instead: with
cfg["alibi"] the scores of head h get + m_h (j - i) (no rotary embedding),
with cfg["act"] == "relu2" the feed-forward is h = max(u, 0)^2 of one up
projection (w_gu then holds only the F "up" rows).  Weights use the [out, in] layout: w_qkv rows are
[Q heads; K heads; V heads], w_gu rows are [gate; up].  Query head h reads
key/value head floor(h * Hkv / H).  RoPE rotates the pairs (i, i + Dh/2) by
angle pos * theta^(-2i/Dh) at in-sequence position pos; theta = 0 disables it.

With per-token masks (``per_token=True``, masks [L, B, S]; see
``oracle/masks.py`` for this reading of the granularity the Tensor
Granularity subsection leaves to future work) the same blocks run on the kept
tokens of each sequence as one shorter sequence: rows in their original
order, rotary angles and ALiBi distances from their original positions, keys
and values of the kept tokens only; a dropped token's row is left unchanged.

The backward is derived by hand from these definitions (chain rule, no
autograd).  Everything is float64, one sequence at a time.
"""

import math

import numpy as np


# --------------------------------------------------------------------------
# building blocks
# --------------------------------------------------------------------------

def rmsnorm(x, gamma, eps):
    """RMSNorm of each row: x / sqrt(mean(x^2) + eps) * gamma.

    Returns (output, normalised rows without gamma, reciprocal rms)."""
    r = 1.0 / np.sqrt(np.mean(x * x, axis=-1) + eps)
    xn = x * r[:, None]
    return xn * gamma, xn, r


def rmsnorm_backward(dy, xn, r, gamma):
    """Gradients of rmsnorm w.r.t. its input rows and gamma.

    With xn = x r and r = (mean(x^2) + eps)^(-1/2):
      d xn = dy * gamma
      dx   = r * (d xn - xn * mean(d xn * xn))
      dgamma = sum over rows of dy * xn."""
    dxn = dy * gamma
    dx = r[:, None] * (dxn - xn * np.mean(dxn * xn, axis=-1, keepdims=True))
    dgamma = np.sum(dy * xn, axis=0)
    return dx, dgamma


def rope_tables(S, Dh, theta):
    """cos, sin of pos * theta^(-2i/Dh), shape [S, Dh/2]."""
    half = Dh // 2
    i = np.arange(half, dtype=np.float64)
    inv_freq = theta ** (-(2.0 * i) / Dh)
    ang = np.arange(S, dtype=np.float64)[:, None] * inv_freq[None, :]
    return np.cos(ang), np.sin(ang)


def rope(t, cos, sin):
    """Rotate pairs (i, i+Dh/2) of every head vector; t is [S, heads, Dh]."""
    half = t.shape[-1] // 2
    a, b = t[..., :half], t[..., half:]
    c, s = cos[:, None, :], sin[:, None, :]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def rope_backward(dt, cos, sin):
    """Transpose of ``rope`` (rotation by the opposite angle)."""
    half = dt.shape[-1] // 2
    a, b = dt[..., :half], dt[..., half:]
    c, s = cos[:, None, :], sin[:, None, :]
    return np.concatenate([a * c + b * s, b * c - a * s], axis=-1)


def kv_head(h, H, Hkv):
    return (h * Hkv) // H


def alibi_slopes(H):
    """Per-head ALiBi slopes (Press et al., "Train Short, Test Long", ICLR
    2022): for a power of two n, the geometric sequence 2^(-8 k / n),
    k = 1..n; otherwise the n0 = 2^floor(log2 H) slopes of that sequence
    followed by every other slope (the 1st, 3rd, ...) of the sequence for
    2 n0, H - n0 of them."""
    def geometric(n):
        return [2.0 ** (-8.0 * k / n) for k in range(1, n + 1)]

    n0 = 2 ** int(math.floor(math.log2(H)))
    if n0 == H:
        return np.array(geometric(H))
    return np.array(geometric(n0) + geometric(2 * n0)[0::2][: H - n0])


def attention_probs(qh, kh, slope=None, pos=None):
    """Causal softmax(q k^T / sqrt(Dh) [+ slope (pos_j - pos_i)]) for one
    head: [S, S].  Rows are in causal order; ``pos`` (default 0 .. S-1) are
    their positions for the ALiBi distance."""
    S, Dh = qh.shape
    sc = (qh @ kh.T) / math.sqrt(Dh)
    if slope is not None:
        pos = np.arange(S, dtype=np.float64) if pos is None else np.asarray(pos, dtype=np.float64)
        sc = sc + slope * (pos[None, :] - pos[:, None])
    causal = np.tril(np.ones((S, S), dtype=bool))
    sc = np.where(causal, sc, -np.inf)
    sc = sc - np.max(sc, axis=1, keepdims=True)
    e = np.exp(sc)
    return e / np.sum(e, axis=1, keepdims=True)


def attention(q, k, v, slopes=None, pos=None):
    """Causal grouped-query attention. q [S,H,Dh], k/v [S,Hkv,Dh] -> [S,H,Dh];
    ``slopes`` [H] adds the ALiBi bias (at positions ``pos``)."""
    S, H, Dh = q.shape
    Hkv = k.shape[1]
    o = np.zeros_like(q)
    for h in range(H):
        j = kv_head(h, H, Hkv)
        P = attention_probs(q[:, h, :], k[:, j, :], None if slopes is None else slopes[h], pos)
        o[:, h, :] = P @ v[:, j, :]
    return o


def attention_backward(do, q, k, v, slopes=None, pos=None):
    """Gradients of ``attention`` w.r.t. q, k, v given d(out) = do.

    Per head, with P the probabilities and c = 1/sqrt(Dh):
      dv += P^T do;  dP = do v^T;  dS = P * (dP - rowsum(dP * P));
      dq = c dS k;   dk += c dS^T q
    (key/value gradients summed over the query heads that share them; the
    ALiBi bias is constant in q and k and only enters through P)."""
    S, H, Dh = q.shape
    Hkv = k.shape[1]
    c = 1.0 / math.sqrt(Dh)
    dq = np.zeros_like(q)
    dk = np.zeros_like(k)
    dv = np.zeros_like(v)
    for h in range(H):
        j = kv_head(h, H, Hkv)
        P = attention_probs(q[:, h, :], k[:, j, :], None if slopes is None else slopes[h], pos)
        doh = do[:, h, :]
        dv[:, j, :] += P.T @ doh
        dP = doh @ v[:, j, :].T
        dS = P * (dP - np.sum(dP * P, axis=1, keepdims=True))
        dq[:, h, :] = c * (dS @ k[:, j, :])
        dk[:, j, :] += c * (dS.T @ q[:, h, :])
    return dq, dk, dv


def relu(x):
    return np.maximum(x, 0.0)


def sigmoid(x):
    with np.errstate(over="ignore"):
        return 1.0 / (1.0 + np.exp(-x))


# --------------------------------------------------------------------------
# one layer, one sequence
# --------------------------------------------------------------------------

def _split_qkv(qkv, cfg):
    S = qkv.shape[0]
    H, Hkv, Dh = cfg["H"], cfg["Hkv"], cfg["Dh"]
    q = qkv[:, : H * Dh].reshape(S, H, Dh)
    k = qkv[:, H * Dh : (H + Hkv) * Dh].reshape(S, Hkv, Dh)
    v = qkv[:, (H + Hkv) * Dh :].reshape(S, Hkv, Dh)
    return q, k, v


def _slopes(cfg):
    return alibi_slopes(cfg["H"]) if cfg.get("alibi") else None


def _positions(S, pos):
    return np.arange(S) if pos is None else np.asarray(pos)


def attn_forward(x, W, cfg, s, rope_cs, pos=None):
    """Attention residual block of a kept sequence: Z = X + s f_attn(X).
    ``pos``: positions of the rows (default 0 .. S-1; the kept tokens'
    original positions with per-token masks)."""
    S = x.shape[0]
    pp = _positions(S, pos)
    xh, xn, r1 = rmsnorm(x, W["g1"], cfg["eps"])
    q, k, v = _split_qkv(xh @ W["w_qkv"].T, cfg)
    if rope_cs is not None:
        cos, sin = rope_cs
        q = rope(q, cos[pp], sin[pp])
        k = rope(k, cos[pp], sin[pp])
    o = attention(q, k, v, _slopes(cfg), pp).reshape(S, -1)
    z = x + s * (o @ W["w_o"].T)
    return z, dict(xh=xh, xn=xn, r1=r1, q=q, k=k, v=v, o=o)


def ffn_forward(z, W, cfg, s):
    """FFN residual block of a kept sequence: X' = Z + s f_ffn(Z), with
    f_ffn = w_d silu(g) u (SwiGLU) or w_d max(u, 0)^2 (squared ReLU)."""
    F = cfg["F"]
    zh, zn, r2 = rmsnorm(z, W["g2"], cfg["eps"])
    gu = zh @ W["w_gu"].T
    if cfg.get("act") == "relu2":
        g, u = None, gu
        h = relu(u) ** 2
    else:
        g, u = gu[:, :F], gu[:, F:]
        h = g * sigmoid(g) * u
    out = z + s * (h @ W["w_d"].T)
    return out, dict(zh=zh, zn=zn, r2=r2, g=g, u=u, h=h)


def layer_forward(x, W, cfg, s, rope_cs):
    """Kept sequence x [S, d] -> X^{l+1}[b] and the values the backward needs."""
    z, ca = attn_forward(x, W, cfg, s, rope_cs)
    out, cf = ffn_forward(z, W, cfg, s)
    return out, {**ca, **cf}


def layer_backward(dout, W, cfg, s, cache, G, rope_cs):
    """d X^{l+1}[b] -> d X^l[b] for a kept sequence; adds into the layer's
    weight gradients G."""
    dz = ffn_backward(dout, W, cfg, s, cache, G)
    return attn_backward(dz, W, cfg, s, cache, G, rope_cs)


def ffn_backward(dout, W, cfg, s, cache, G):
    """d X'[b] -> d Z[b] through the FFN block; adds into G."""
    c = cache
    # out = z + s * (h w_d^T), h = silu(g) u.
    dy = s * dout
    G["w_d"] += dy.T @ c["h"]
    dh = dy @ W["w_d"]
    if cfg.get("act") == "relu2":
        dgu = dh * 2.0 * relu(c["u"])      # d/du max(u, 0)^2 = 2 max(u, 0)
    else:
        sg = sigmoid(c["g"])
        dg = dh * c["u"] * sg * (1.0 + c["g"] * (1.0 - sg))
        du = dh * c["g"] * sg
        dgu = np.concatenate([dg, du], axis=1)
    G["w_gu"] += dgu.T @ c["zh"]
    dzh = dgu @ W["w_gu"]
    dz_norm, dg2 = rmsnorm_backward(dzh, c["zn"], c["r2"], W["g2"])
    G["g2"] += dg2
    return dout + dz_norm


def attn_backward(dz, W, cfg, s, cache, G, rope_cs, pos=None):
    """d Z[b] -> d X[b] through the attention block; adds into G."""
    S = dz.shape[0]
    pp = _positions(S, pos)
    H, Dh = cfg["H"], cfg["Dh"]
    c = cache
    # z = x + s * (o w_o^T).
    da = s * dz
    G["w_o"] += da.T @ c["o"]
    do = (da @ W["w_o"]).reshape(S, H, Dh)
    dq, dk, dv = attention_backward(do, c["q"], c["k"], c["v"], _slopes(cfg), pp)
    if rope_cs is not None:
        cos, sin = rope_cs
        dq = rope_backward(dq, cos[pp], sin[pp])
        dk = rope_backward(dk, cos[pp], sin[pp])
    dqkv = np.concatenate([dq.reshape(S, -1), dk.reshape(S, -1), dv.reshape(S, -1)], axis=1)
    G["w_qkv"] += dqkv.T @ c["xh"]
    dxh = dqkv @ W["w_qkv"]
    dx_norm, dg1 = rmsnorm_backward(dxh, c["xn"], c["r1"], W["g1"])
    G["g1"] += dg1
    return dz + dx_norm


# --------------------------------------------------------------------------
# the stack
# --------------------------------------------------------------------------

WEIGHT_NAMES = ("w_qkv", "w_o", "w_gu", "w_d", "g1", "g2")


def _layer(layers, l):
    """Weights of layer l as float64 arrays (``layers`` is a list or a callable)."""
    W = layers(l) if callable(layers) else layers[l]
    return {n: np.asarray(W[n], dtype=np.float64) for n in WEIGHT_NAMES}


def _rope_cs(cfg, S):
    theta = cfg.get("rope_theta", 0.0)
    if not theta or cfg.get("alibi"):
        return None
    return rope_tables(S, cfg["Dh"], theta)


def _branch_masks(masks):
    """(attention mask [L, B], FFN mask [L, B]) from a layer mask [L, B]
    (both blocks share it, layer granularity) or a sub-layer pair [2, L, B]
    (independent M_attn and M_ffn, Model Granularity subsection)."""
    masks = np.asarray(masks)
    if masks.ndim == 3:
        return masks[0], masks[1]
    return masks, masks


def _token_branch_masks(masks):
    masks = np.asarray(masks)
    if masks.ndim == 4:
        return masks[0], masks[1]
    return masks, masks


def stack_forward_tokens(x, layers, cfg, masks, scales):
    """Per-token masks [L, B, S] or [2, L, B, S]: each block runs on the kept
    tokens of each sequence (original order and positions) and updates only
    their rows."""
    X = np.array(x, dtype=np.float64, copy=True)
    B, S, _ = X.shape
    ma, mf = _token_branch_masks(masks)
    L = ma.shape[0]
    rope_cs = _rope_cs(cfg, S)
    caches = [[None] * B for _ in range(L)]
    for l in range(L):
        if not (ma[l].any() or mf[l].any()):
            continue
        W = _layer(layers, l)
        for b in range(B):
            c = {}
            ka = np.nonzero(ma[l, b])[0]
            if ka.size:
                X[b, ka], ca = attn_forward(X[b, ka], W, cfg, scales[l], rope_cs, pos=ka)
                c.update(ca)
            kf = np.nonzero(mf[l, b])[0]
            if kf.size:
                X[b, kf], cf = ffn_forward(X[b, kf], W, cfg, scales[l])
                c.update(cf)
            c.update(ka=ka, kf=kf)
            caches[l][b] = c
    return X, caches


def stack_backward_tokens(dy, layers, cfg, masks, scales, caches):
    """Backward of ``stack_forward_tokens``: a dropped token's gradient
    passes through the block unchanged; weight gradients sum over the kept
    tokens only."""
    dX = np.array(dy, dtype=np.float64, copy=True)
    B, S, _ = dX.shape
    ma, mf = _token_branch_masks(masks)
    L = ma.shape[0]
    rope_cs = _rope_cs(cfg, S)
    grads = [None] * L
    for l in reversed(range(L)):
        W = _layer(layers, l) if (ma[l].any() or mf[l].any()) else None
        G = {n: np.zeros(shape_of(cfg, n)) for n in WEIGHT_NAMES}
        for b in range(B):
            c = caches[l][b]
            if c is None:
                continue
            if c["kf"].size:
                dX[b, c["kf"]] = ffn_backward(dX[b, c["kf"]], W, cfg, scales[l], c, G)
            if c["ka"].size:
                dX[b, c["ka"]] = attn_backward(dX[b, c["ka"]], W, cfg, scales[l], c, G, rope_cs, pos=c["ka"])
        grads[l] = G
    return dX, grads


def stack_forward(x, layers, cfg, masks, scales, per_token=False):
    """x [B, S, d] -> (X^L, caches).  masks [L, B] or [2, L, B] (1 = keep),
    scales [L]; with ``per_token`` masks [L, B, S] or [2, L, B, S]."""
    if per_token:
        return stack_forward_tokens(x, layers, cfg, masks, scales)
    X = np.array(x, dtype=np.float64, copy=True)
    B, S, _ = X.shape
    ma, mf = _branch_masks(masks)
    L = ma.shape[0]
    rope_cs = _rope_cs(cfg, S)
    caches = [[None] * B for _ in range(L)]
    for l in range(L):
        if not (ma[l].any() or mf[l].any()):
            continue
        W = _layer(layers, l)
        for b in range(B):
            c = {}
            if ma[l, b]:
                X[b], ca = attn_forward(X[b], W, cfg, scales[l], rope_cs)
                c.update(ca)
            if mf[l, b]:
                X[b], cf = ffn_forward(X[b], W, cfg, scales[l])
                c.update(cf)
            if c:
                caches[l][b] = c
    return X, caches


def stack_forward_eval(x, layers, cfg, execute, r_eval=None):
    """Depth-elastic inference, Eq. (transformer_layer_dropout_eval): every
    sequence runs Z = X + r_eval f_attn(X), X' = Z + r_eval f_ffn(Z) on each
    layer l with execute[l] = 1 and skips the others (early exit at l' runs
    layers 0 .. l'-1; intermediate skipping any other pattern, Inference
    Optimizations section).  r_eval defaults to 1, the paper's choice."""
    X = np.array(x, dtype=np.float64, copy=True)
    B, S, _ = X.shape
    rope_cs = _rope_cs(cfg, S)
    for l in range(len(execute)):
        if not execute[l]:
            continue
        W = _layer(layers, l)
        r = 1.0 if r_eval is None else float(r_eval[l])
        for b in range(B):
            X[b], _ = layer_forward(X[b], W, cfg, r, rope_cs)
    return X


def stack_backward(dy, layers, cfg, masks, scales, caches, per_token=False):
    """d X^L -> (d X^0, per-layer weight gradients).

    Dropped sequences pass their gradient through unchanged; a block's weight
    gradients sum over its kept sequences only (zero if none is kept)."""
    if per_token:
        return stack_backward_tokens(dy, layers, cfg, masks, scales, caches)
    dX = np.array(dy, dtype=np.float64, copy=True)
    B, S, _ = dX.shape
    ma, mf = _branch_masks(masks)
    L = ma.shape[0]
    rope_cs = _rope_cs(cfg, S)
    grads = [None] * L
    for l in reversed(range(L)):
        W = _layer(layers, l) if (ma[l].any() or mf[l].any()) else None
        G = {n: np.zeros(shape_of(cfg, n)) for n in WEIGHT_NAMES}
        for b in range(B):
            if mf[l, b]:
                dX[b] = ffn_backward(dX[b], W, cfg, scales[l], caches[l][b], G)
            if ma[l, b]:
                dX[b] = attn_backward(dX[b], W, cfg, scales[l], caches[l][b], G, rope_cs)
        grads[l] = G
    return dX, grads


def shape_of(cfg, name):
    d, H, Hkv, Dh, F = cfg["d"], cfg["H"], cfg["Hkv"], cfg["Dh"], cfg["F"]
    return {
        "w_qkv": ((H + 2 * Hkv) * Dh, d),
        "w_o": (d, H * Dh),
        "w_gu": ((F if cfg.get("act") == "relu2" else 2 * F), d),
        "w_d": (d, F),
        "g1": (d,),
        "g2": (d,),
    }[name]
