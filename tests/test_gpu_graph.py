"""A whole step (ld_forward + ld_backward) enqueues only stream-ordered work,
so it can be captured into a CUDA graph and replayed: the replay reproduces
the eager step: outputs bit for bit; input and weight gradients up to the
order of the float32 dQ reductions, whose rounding to bf16 can move by an ulp
and feeds dX and the w_qkv gradient (checked to 1e-2 of the tensor's max)."""

import pytest
import torch

import paper_2609_05275_gb300 as P
from paper_2609_05275_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name", ["tiny", "gpt2"])
def test_step_replays_from_cuda_graph(name):
    cfg = dict(synth.CONFIGS[name])
    if name == "gpt2":
        cfg.update(L=3, B=4)
    sched = dict(dist="ild", p_max=0.5, time="const", seed=4)
    st = P.LayerDropStack(cfg, sched)
    layers = synth.stack_weights(cfg, seed=0, device="cuda")
    wtab = P.weight_table(layers)
    grads = [{n: torch.zeros(v.shape, device="cuda", dtype=torch.float32) for n, v in W.items()} for W in layers]
    gtab = P.grad_table(grads)
    x0 = synth.activations(cfg, device="cuda")
    dy0 = synth.upstream_grad(cfg, device="cuda")
    x, dx = x0.clone(), dy0.clone()
    st.forward(5, wtab, x)  # eager step (also does the one-time per-kernel set-up)
    st.backward(wtab, dx, gtab)
    torch.cuda.synchronize()
    st.sync()
    ref_x, ref_dx = x.clone(), dx.clone()
    ref_g = [{n: g.clone() for n, g in G.items()} for G in grads]

    graph = torch.cuda.CUDAGraph()
    x.copy_(x0)
    dx.copy_(dy0)
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(stream):
        with torch.cuda.graph(graph, stream=stream):
            st.forward(5, wtab, x)
            st.backward(wtab, dx, gtab)
    torch.cuda.current_stream().wait_stream(stream)
    for _ in range(2):
        x.copy_(x0)
        dx.copy_(dy0)
        for G in grads:
            for g in G.values():
                g.fill_(float("nan"))
        graph.replay()
        torch.cuda.synchronize()
        assert torch.equal(x, ref_x)
        assert (dx.float() - ref_dx.float()).abs().max().item() <= 2e-2 * ref_dx.float().abs().max().item() + 1e-3
        for G, R in zip(grads, ref_g):
            for n in G:
                assert (G[n] - R[n]).abs().max().item() <= 1e-2 * R[n].abs().max().item() + 1e-6, n
    st.close()
