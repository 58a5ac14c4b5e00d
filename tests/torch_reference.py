"""An independent dense decoder layer in PyTorch (float64, CPU), used only to
pin the oracle.

It is written with library routines that the oracle does not use:
``torch.nn.functional.rms_norm``, ``scaled_dot_product_attention`` with a
causal mask, complex multiplication for the rotary embedding, ``F.silu``, and
autograd for every gradient.  A mistake in the oracle's hand-written forward
or hand-derived backward (a dropped term, a sign, a transposed operand, a
wrong key/value head) shows up as a mismatch with this module.
"""

import torch
import torch.nn.functional as F


def _rope_complex(t, theta, pos=None):
    """t [S, heads, Dh]; pairs (i, i + Dh/2) rotated as complex numbers by
    angle pos * freq (pos defaults to 0 .. S-1)."""
    S, nh, Dh = t.shape
    half = Dh // 2
    freqs = 1.0 / (theta ** (torch.arange(0, Dh, 2, dtype=torch.float64) / Dh))
    p = torch.arange(S, dtype=torch.float64) if pos is None else torch.as_tensor(pos, dtype=torch.float64)
    ang = torch.outer(p, freqs)
    rot = torch.polar(torch.ones_like(ang), ang)[:, None, :]
    c = torch.complex(t[..., :half], t[..., half:]) * rot
    return torch.cat([c.real, c.imag], dim=-1)


def dense_layer(x, W, cfg, slopes=None, pos=None):
    """f for one sequence x [S, d] at rate 0 and scale 1: returns (attn, ffn)
    callables so that masks and scales can be composed outside.  With
    cfg["alibi"] the per-head ``slopes`` enter SDPA as an additive float mask
    m_h (j - i) next to -inf above the diagonal; cfg["act"] == "relu2" selects
    the squared-ReLU feed-forward.  ``pos`` (increasing; default 0 .. S-1)
    are the rows' positions for the rotary angles and ALiBi distances."""
    H, Hkv, Dh, Fh = cfg["H"], cfg["Hkv"], cfg["Dh"], cfg["F"]
    eps, theta = cfg["eps"], cfg.get("rope_theta", 0.0)
    S = x.shape[0]
    alibi = cfg.get("alibi", False)
    if alibi:
        theta = 0.0
        pp = torch.arange(S, dtype=torch.float64) if pos is None else torch.as_tensor(pos, dtype=torch.float64)
        rel = pp[None, :] - pp[:, None]
        bias = torch.as_tensor(slopes, dtype=torch.float64)[:, None, None] * rel[None]
        bias = bias.masked_fill(rel[None] > 0, float("-inf"))

    def f_attn(xx):
        xh = F.rms_norm(xx, (xx.shape[-1],), weight=W["g1"], eps=eps)
        qkv = xh @ W["w_qkv"].T
        q = qkv[:, : H * Dh].view(S, H, Dh)
        k = qkv[:, H * Dh : (H + Hkv) * Dh].view(S, Hkv, Dh)
        v = qkv[:, (H + Hkv) * Dh :].view(S, Hkv, Dh)
        if theta:
            q, k = _rope_complex(q, theta, pos), _rope_complex(k, theta, pos)
        rep = H // Hkv
        k = k.repeat_interleave(rep, dim=1)
        v = v.repeat_interleave(rep, dim=1)
        qq, kk, vv = q.transpose(0, 1)[None], k.transpose(0, 1)[None], v.transpose(0, 1)[None]
        if alibi:
            o = F.scaled_dot_product_attention(qq, kk, vv, attn_mask=bias[None])
        else:
            o = F.scaled_dot_product_attention(qq, kk, vv, is_causal=True)
        o = o[0].transpose(0, 1).reshape(S, H * Dh)
        return o @ W["w_o"].T

    def f_ffn(zz):
        zh = F.rms_norm(zz, (zz.shape[-1],), weight=W["g2"], eps=eps)
        gu = zh @ W["w_gu"].T
        if cfg.get("act") == "relu2":
            return F.relu(gu).square() @ W["w_d"].T
        return (F.silu(gu[:, :Fh]) * gu[:, Fh:]) @ W["w_d"].T

    return f_attn, f_ffn


def masked_stack(x, layers, cfg, masks, scales, slopes=None):
    """Stack with per-sequence masks, composed from dense layers:
    z = x + s M_attn f_attn(x), x' = z + s M_ffn f_ffn(z), where masks is
    [L, B] (M_attn = M_ffn = masks, layer granularity) or [2, L, B]
    (M_attn = masks[0], M_ffn = masks[1], sub-layer granularity)."""
    ma, mf = (masks[0], masks[1]) if masks.ndim == 3 else (masks, masks)
    B = x.shape[0]
    outs = []
    for b in range(B):
        xb = x[b]
        for l in range(ma.shape[0]):
            f_attn, f_ffn = dense_layer(xb, layers[l], cfg, slopes)
            s = float(scales[l])
            zb = xb + s * f_attn(xb) if ma[l, b] else xb
            xb = zb + s * f_ffn(zb) if mf[l, b] else zb
        outs.append(xb)
    return torch.stack(outs)


def token_masked_stack(x, layers, cfg, masks, scales, slopes=None):
    """Stack with per-token masks [L, B, S] (or [2, L, B, S] for separate
    attention / FFN masks), composed from dense layers applied to each
    sequence's kept tokens as one shorter sequence at their original
    positions; the other rows are left as they are."""
    masks = torch.as_tensor(masks)
    ma, mf = (masks[0], masks[1]) if masks.ndim == 4 else (masks, masks)
    outs = []
    for b in range(x.shape[0]):
        xb = x[b]
        for l in range(ma.shape[0]):
            s = float(scales[l])
            ka = torch.nonzero(ma[l, b]).flatten()
            if ka.numel():
                f_attn, _ = dense_layer(xb[ka], layers[l], cfg, slopes, pos=ka)
                xb = torch.index_add(xb, 0, ka, s * f_attn(xb[ka]))
            kf = torch.nonzero(mf[l, b]).flatten()
            if kf.numel():
                _, f_ffn = dense_layer(xb[kf], layers[l], cfg, slopes, pos=kf)
                xb = torch.index_add(xb, 0, kf, s * f_ffn(xb[kf]))
        outs.append(xb)
    return torch.stack(outs)


def to_torch_layers(layers, requires_grad=False):
    out = []
    for W in layers:
        out.append({n: torch.tensor(W[n], dtype=torch.float64, requires_grad=requires_grad)
                    for n in ("w_qkv", "w_o", "w_gu", "w_d", "g1", "g2")})
    return out
