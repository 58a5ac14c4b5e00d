"""Data-parallel sharding on one GPU: the batch run as two shards one after
the other (b_offset 0 and B/2) gives bit-identical masks and outputs, input
gradients within the bf16 tolerance (dQ is summed over key tiles with float
atomics, so its last bits depend on the order), and shard weight gradients
that sum to the full batch's."""

import numpy as np
import pytest
import torch

from paper_2609_05275_gb300 import synth
import paper_2609_05275_gb300 as P

pytestmark = pytest.mark.gpu


def _run(cfg, sched, x, dy, layers, b_offset):
    st = P.LayerDropStack(cfg, sched, b_offset=b_offset)
    try:
        wtab = P.weight_table(layers)
        xx, dd = x.clone(), dy.clone()
        grads = [{n: torch.empty(v.shape, device="cuda", dtype=torch.float32) for n, v in W.items()} for W in layers]
        st.forward(7, wtab, xx)
        st.backward(wtab, dd, P.grad_table(grads))
        torch.cuda.synchronize()
        st.sync()
        return xx, dd, grads, st.masks()
    finally:
        st.close()


@pytest.mark.parametrize("name", ["tiny", "gpt2"])
def test_two_shards_equal_full_batch(name):
    cfg = dict(synth.CONFIGS[name])
    if name == "gpt2":
        cfg.update(L=4, B=8)
    sched = dict(dist="ild", p_max=0.6, time="const", seed=3)
    layers = synth.stack_weights(cfg, seed=0, device="cuda")
    x = synth.activations(cfg, seed=0, device="cuda").view(cfg["B"] * cfg["S"], -1)
    dy = synth.upstream_grad(cfg, device="cuda").view(cfg["B"] * cfg["S"], -1)
    full = _run(cfg, sched, x, dy, layers, 0)
    half = cfg["B"] // 2
    rows = half * cfg["S"]
    scfg = dict(cfg, B=half)
    s0 = _run(scfg, sched, x[:rows], dy[:rows], layers, 0)
    s1 = _run(scfg, sched, x[rows:], dy[rows:], layers, half)
    assert np.array_equal(np.concatenate([s0[3][0], s1[3][0]], axis=1), full[3][0])
    assert torch.equal(torch.cat([s0[0], s1[0]]), full[0])
    dxs, dxf = torch.cat([s0[1], s1[1]]).float(), full[1].float()
    assert (dxs - dxf).abs().max().item() <= 2e-2 * dxf.abs().max().item() + 1e-3
    for l in range(cfg["L"]):
        for n in full[2][l]:
            ref = full[2][l][n]
            got = s0[2][l][n] + s1[2][l][n]
            assert (got - ref).abs().max().item() <= 2e-2 * ref.abs().max().item() + 1e-3, (l, n)
