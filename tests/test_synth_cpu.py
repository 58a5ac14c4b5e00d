"""The seeded synthetic input recipe (paper_2609_05275_gb300/synth.py):
shapes of every workload, the stated distributions, the depth-scaled init
of the residual output projections, bf16-representable values and
reproducibility of each tensor from (seed, tag, layer) alone."""

import math

import pytest
import torch

from paper_2609_05275_gb300 import synth

SMALL_DEEP = dict(L=8, d=256, H=4, Hkv=2, Dh=64, F=512, B=2, S=128, eps=1e-6, rope_theta=1e4, alpha=1.0,
                  init="depth_scaled")


@pytest.mark.parametrize("name", sorted(synth.CONFIGS))
def test_weight_shapes(name):
    cfg = synth.CONFIGS[name]
    d, H, Hkv, Dh, F = cfg["d"], cfg["H"], cfg["Hkv"], cfg["Dh"], cfg["F"]
    s = synth.weight_shapes(cfg)
    assert s["w_qkv"] == ((H + 2 * Hkv) * Dh, d) and s["w_o"] == (d, H * Dh) and s["w_d"] == (d, F)
    assert s["w_gu"] == ((F if cfg.get("act") == "relu2" else 2 * F), d)
    assert s["g1"] == s["g2"] == (d,)
    assert H % Hkv == 0


def test_distributions_and_depth_scaled_init():
    W = synth.layer_weights(SMALL_DEEP, 3, seed=5)
    for n in ("w_qkv", "w_gu"):
        assert W[n].float().std().item() == pytest.approx(0.02, rel=0.05)
    for n in ("w_o", "w_d"):
        assert W[n].float().std().item() == pytest.approx(0.02 / math.sqrt(2 * SMALL_DEEP["L"]), rel=0.05)
    assert torch.equal(W["g1"], torch.ones_like(W["g1"])) and torch.equal(W["g2"], torch.ones_like(W["g2"]))
    plain = dict(SMALL_DEEP)
    plain.pop("init")
    assert synth.layer_weights(plain, 3, seed=5)["w_o"].float().std().item() == pytest.approx(0.02, rel=0.05)
    x = synth.activations(SMALL_DEEP, seed=1).float()
    dy = synth.upstream_grad(SMALL_DEEP).float()
    for t in (x, dy):
        assert t.shape == (2, 128, 256)
        assert abs(t.mean().item()) < 0.02 and t.std().item() == pytest.approx(1.0, rel=0.02)
    g = synth.layer_weights(SMALL_DEEP, 0, gamma_noise=0.1)["g1"].float()
    assert (g - 1).std().item() == pytest.approx(0.1, rel=0.2)


def test_values_are_bf16_and_reproducible():
    a = synth.layer_weights(SMALL_DEEP, 2, seed=7, dtype=torch.float32)
    b = synth.layer_weights(SMALL_DEEP, 2, seed=7)
    for n in a:
        assert torch.equal(a[n], b[n].float())  # the float32 copy holds bf16 values exactly
    c = synth.layer_weights(SMALL_DEEP, 2, seed=7)
    assert all(torch.equal(b[n], c[n]) for n in b)
    d = synth.layer_weights(SMALL_DEEP, 3, seed=7)
    e = synth.layer_weights(SMALL_DEEP, 2, seed=8)
    assert not torch.equal(b["w_qkv"], d["w_qkv"]) and not torch.equal(b["w_qkv"], e["w_qkv"])
    # each tensor has its own stream: one layer regenerates alone, equal to the stack's
    st = synth.stack_weights(SMALL_DEEP, seed=7)
    assert all(torch.equal(st[2][n], b[n]) for n in b)
    x1 = synth.activations(SMALL_DEEP, seed=1, B=1)
    x2 = synth.activations(SMALL_DEEP, seed=1)
    assert torch.equal(x1[0], x2[0])
