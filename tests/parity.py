"""Helpers shared by the parity tests: run the CUDA stack through the C ABI
and the oracle on the same seeded inputs, and compare per tensor.

Tolerances:
  bf16 path      max|gpu - ref| <= 2e-2 * max|ref| + 1e-3 (per tensor)
  float32 path   max|gpu - ref| <= 1e-5 * max|ref|        (per tensor)
"""

import numpy as np
import torch

import paper_2609_05275_gb300 as P
from paper_2609_05275_gb300 import synth
from oracle import masks as OM
from oracle import schedule as OS
from oracle import stack as OK

BF16_REL, BF16_ABS = 2e-2, 1e-3
F32_REL = 1e-5


def oracle_sched(sched):
    """The oracle's schedule dict for a workload schedule."""
    d = dict(dist=sched["dist"], p_max=sched.get("p_max", 0.0), p_explicit=sched.get("p_explicit"),
             time=sched.get("time", "const"), T=sched.get("T"), ramp=sched.get("ramp"))
    return d


def oracle_masks(cfg, sched, step, granularity="per_sequence", sublayer=False):
    rates = OS.layer_rates(oracle_sched(sched), cfg["L"], step)
    thr = [OS.drop_threshold(p) for p in rates]
    scales = [OS.residual_scale(p, cfg.get("alpha", 1.0)) for p in rates]
    gran = {"per_sequence": OM.PER_SEQUENCE, "per_batch": OM.PER_BATCH, "per_shard": OM.PER_SHARD,
            "per_token": OM.PER_TOKEN}[granularity]
    mask = OM.draw_masks(sched.get("seed", 0), step, thr, cfg["B"], gran, sublayer=sublayer, S=cfg["S"])
    return mask, thr, scales


def check_close(name, got, ref, fp32=False):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (name, got.shape, ref.shape)
    err = float(np.max(np.abs(got - ref))) if got.size else 0.0
    mref = float(np.max(np.abs(ref))) if ref.size else 0.0
    bound = F32_REL * mref if fp32 else BF16_REL * mref + BF16_ABS
    assert np.isfinite(got).all(), f"{name}: non-finite values"
    assert err <= bound, f"{name}: max|gpu-ref| = {err:.3e} > {bound:.3e} (max|ref| = {mref:.3e})"
    return err, mref


def to_np(t):
    return t.detach().float().cpu().double().numpy() if t.dtype != torch.float64 else t.detach().cpu().numpy()


def gpu_run(cfg, sched, step, layers_dev, x_dev, dy_dev, granularity="per_sequence", fp32_debug=False,
            backward=True, sublayer=False):
    """Forward (+ backward) through the C ABI.  Returns (out, dX, grads, masks)."""
    st = P.LayerDropStack(cfg, sched, granularity=granularity, fp32_debug=fp32_debug, sublayer=sublayer)
    try:
        wtab = P.weight_table(layers_dev)
        x = x_dev.clone()
        st.forward(step, wtab, x)
        dx, grads = None, None
        if backward:
            dx = dy_dev.clone()
            grads = [{n: torch.full(v.shape, float("nan"), device=v.device, dtype=torch.float32)
                      for n, v in W.items()} for W in layers_dev]
            st.backward(wtab, dx, P.grad_table(grads))
        torch.cuda.synchronize()
        st.sync()
        masks = st.masks()
        return x, dx, grads, masks
    finally:
        st.close()


def oracle_run(cfg, sched, step, layers_host, x_host, dy_host, granularity="per_sequence", rows=None,
               seqs=None, sublayer=False):
    """The oracle on (optionally) the first `rows` rows of the sequences
    `seqs`; returns (out, dX, grads, mask)."""
    mask, thr, scales = oracle_masks(cfg, sched, step, granularity, sublayer)
    x = x_host.double().numpy()
    dy = dy_host.double().numpy()
    mk = mask
    tok = granularity == "per_token"
    if seqs is not None:
        x, dy, mk = x[seqs], dy[seqs], (mask[..., seqs, :] if tok else mask[..., seqs])
    if rows is not None:
        x, dy = x[:, :rows], dy[:, :rows]
        if tok:
            mk = mk[..., :rows]

    def layer(l):
        return {n: v.double().numpy() for n, v in layers_host[l].items()}

    out, caches = OK.stack_forward(x, layer, cfg, mk, scales, per_token=tok)
    dX, grads = OK.stack_backward(dy, layer, cfg, mk, scales, caches, per_token=tok)
    return out, dX, grads, mask
