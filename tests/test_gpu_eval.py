"""Depth-elastic inference forward (Eq. transformer_layer_dropout_eval)
through the C ABI against the oracle: early exit, intermediate layer
skipping, r_eval != 1, every layer skipped (identity), batch-1 / short-S
shapes, the paper's architecture, and a workspace of exactly
ld_eval_workspace_size bytes."""

import numpy as np
import pytest
import torch

import paper_2609_05275_gb300 as P
from paper_2609_05275_gb300 import synth
from parity import check_close, to_np
from oracle import stack as OK

pytestmark = pytest.mark.gpu


def _eval(cfg, execute, r_eval=None, fp32=False, seed=0):
    dtype = torch.float32 if fp32 else torch.bfloat16
    host = synth.stack_weights(cfg, seed=seed, gamma_noise=0.1)
    x = synth.activations(cfg, seed=seed)
    # weights of skipped layers are not handed over at all
    dev = [({n: v.to(dtype).cuda() for n, v in W.items()} if e else None) for W, e in zip(host, execute)]
    st = P.LayerDropStack(cfg, dict(dist="uniform", p_max=0.0, seed=1), fp32_debug=fp32)
    try:
        nb = P.ld_eval_workspace_size(st.h)
        st.workspace = torch.empty(nb, dtype=torch.uint8, device="cuda")  # the evaluation minimum only
        xd = x.to(dtype).cuda()
        out = xd.clone()
        st.forward_eval(execute, P.weight_table(dev), out, r_eval)
        torch.cuda.synchronize()
        st.sync()
    finally:
        st.close()

    def layer(l):
        return {n: v.double().numpy() for n, v in host[l].items()}

    ref = OK.stack_forward_eval(x.double().numpy(), layer, cfg, execute, r_eval)
    check_close("eval out", to_np(out), ref, fp32)
    return out, xd


@pytest.mark.parametrize("fp32", [True, False], ids=["fp32", "bf16"])
def test_early_exit_and_skipping(fp32):
    cfg = dict(synth.CONFIGS["tiny"], L=4, H=4, Hkv=2)
    _eval(cfg, [1, 1, 1, 1], fp32=fp32)
    _eval(cfg, [1, 1, 0, 0], fp32=fp32)                             # early exit at l' = 2
    _eval(cfg, [1, 0, 1, 0], [1.0, 1.0, 0.5, 1.0], fp32=fp32)       # alternate layers, r_eval = 0.5 on one
    out, xd = _eval(cfg, [0, 0, 0, 0], fp32=fp32)                   # nothing executed: identity
    assert torch.equal(out, xd)


@pytest.mark.parametrize("cfg", [
    dict(L=3, d=512, H=4, Hkv=1, Dh=128, F=1024, B=1, S=128, eps=1e-6, rope_theta=5e5, alpha=1.0),   # batch 1
    dict(L=3, d=256, H=4, Hkv=2, Dh=64, F=512, B=2, S=64, eps=1e-6, rope_theta=1e4, alpha=1.0),      # S = 64
    dict(L=3, d=512, H=4, Hkv=4, Dh=128, F=2048, B=2, S=1024, eps=1e-6, rope_theta=0.0, alpha=1.0,
         alibi=True, act="relu2"),                                                                # paper arch
], ids=["b1-s128", "b2-s64", "paper-arch"])
def test_decode_shapes_and_paper_arch(cfg):
    _eval(cfg, [1, 0, 1])
    _eval(cfg, [1, 1, 0], [1.0, 0.8, 1.0])


def test_eval_matches_training_forward_at_p0():
    # all layers at r_eval = 1 is the training forward at p = 0 (scale 1), bit for bit
    cfg = dict(synth.CONFIGS["gpt2"], L=3, B=2)
    layers = synth.stack_weights(cfg, seed=0, device="cuda")
    x = synth.activations(cfg, device="cuda")
    wtab = P.weight_table(layers)
    st = P.LayerDropStack(cfg, dict(dist="uniform", p_max=0.0, seed=1))
    try:
        a, b = x.clone(), x.clone()
        st.forward(0, wtab, a)
        st.forward_eval([1, 1, 1], wtab, b)
        torch.cuda.synchronize()
        st.sync()
        assert torch.equal(a, b)
        # the evaluation forward leaves no state for a backward
        with pytest.raises(P.LdError):
            st.backward(wtab, b, P.grad_table([{n: torch.zeros(v.shape, device="cuda") for n, v in W.items()}
                                               for W in layers]))
    finally:
        st.close()


@pytest.mark.parametrize("fp32", [True, False], ids=["fp32", "bf16"])
def test_eval_on_per_token_handle(fp32):
    # the evaluation forward runs whole sequences whatever the handle's
    # granularity: a per-token handle gives the per-sequence handle's output
    # bit for bit (its larger mask tables hold the per-sequence lists)
    cfg = (dict(synth.CONFIGS["tiny"], L=3) if fp32 else
           dict(L=3, d=256, H=2, Hkv=1, Dh=128, F=512, B=3, S=256, eps=1e-6, rope_theta=1e4, alpha=1.0))
    dtype = torch.float32 if fp32 else torch.bfloat16
    host = synth.stack_weights(cfg, seed=4, gamma_noise=0.1)
    dev = [{n: v.to(dtype).cuda() for n, v in W.items()} for W in host]
    x = synth.activations(cfg, seed=4).to(dtype).cuda()
    outs = []
    for gran in ("per_sequence", "per_token"):
        st = P.LayerDropStack(cfg, dict(dist="uniform", p_max=0.0, seed=1), granularity=gran, fp32_debug=fp32)
        try:
            out = x.clone()
            st.forward_eval([1, 0, 1], P.weight_table(dev), out)
            torch.cuda.synchronize()
            st.sync()
            outs.append(out)
        finally:
            st.close()
    assert torch.equal(outs[0], outs[1])
