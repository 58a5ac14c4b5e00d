"""Seeded synthetic inputs and the named workload shapes.

This module generates inputs only; it holds none of the method's arithmetic
(no schedule, no mask draw, no layer math).  Both the CUDA path and the CPU
oracle take their inputs from here.

Recipe (the paper trains on a private corpus on Cerebras CS-3; token values
do not change the work done, so activations stand in for embedded tokens):
  * activations x ~ N(0, 1) drawn in float32, rounded to bf16;
  * weights N(0, 0.02) per matrix, RMSNorm gains gamma = 1 (optionally
    1 + N(0, 0.1) to exercise the gain gradient), rounded to bf16; workloads
    with init "depth_scaled" draw the residual output projections (w_o, w_d)
    with std 0.02 / sqrt(2 L), the depth-scaled init of deep pre-norm
    decoders, so that the residual branches do not grow with depth;
  * upstream gradient dY ~ N(0, 1) in float32, rounded to bf16.
Every tensor comes from its own ``torch.Generator`` seeded from (seed, tag,
layer), so any one of them can be regenerated alone.
"""

import torch

# Workload shapes: L layers, model width d, H query heads of size Dh, Hkv
# key/value heads, SwiGLU hidden F, batch B of sequences of length S.
CONFIGS = {
    "tiny": dict(L=2, d=128, H=4, Hkv=4, Dh=32, F=512, B=8, S=64, eps=1e-6, rope_theta=1e4, alpha=1.0),
    "gpt2": dict(L=12, d=768, H=12, Hkv=12, Dh=64, F=2048, B=16, S=1024, eps=1e-6, rope_theta=1e4, alpha=1.0),
    "1.3b": dict(L=24, d=2048, H=16, Hkv=16, Dh=128, F=5632, B=8, S=2048, eps=1e-6, rope_theta=1e4, alpha=1.0,
                 init="depth_scaled"),
    "llama8b": dict(L=32, d=4096, H=32, Hkv=8, Dh=128, F=14336, B=4, S=4096, eps=1e-6, rope_theta=5e5, alpha=1.0,
                    init="depth_scaled"),
    # the paper's own architecture (Methodology section; model table): ALiBi
    # position biases, squared-ReLU feed-forward of width 8 d, 3.9B shape;
    # batch and sequence length chosen here (16384 tokens like the others)
    "paper-3.9b": dict(L=40, d=2048, H=16, Hkv=16, Dh=128, F=16384, B=8, S=2048, eps=1e-6, rope_theta=0.0,
                       alpha=1.0, alibi=True, act="relu2", init="depth_scaled"),
}

# Drop-rate schedules the workloads name (distribution x time schedule, seed).
SCHEDULES = {
    "tiny": dict(dist="explicit", p_max=0.0, p_explicit=[0.0, 0.5], time="const", seed=1),
    "gpt2": dict(dist="ild", p_max=0.2, time="const", seed=1),
    "1.3b": dict(dist="ild", p_max=0.3, time="ramp", ramp=(0, 1000, 0.0, 1.0), seed=1),
    "llama8b": dict(dist="ild", p_max=0.4, time="const", seed=1),
    "paper-3.9b": dict(dist="ild", p_max=0.4, time="const", seed=1),
}

# Steps at which each workload is run (the 1.3B ramp is sampled at 0/500/2000).
STEPS = {"tiny": [0], "gpt2": [0], "1.3b": [0, 500, 2000], "llama8b": [0], "paper-3.9b": [0]}

# Sweep on the 1.3B shape: p_max x distribution x granularity x seeds.
SWEEP = dict(base="1.3b", p_max=[0.0, 0.1, 0.2, 0.3, 0.5], dist=["ild", "uniform"],
             granularity=["per_sequence", "per_batch", "per_token"], seeds=list(range(1, 21)))

_TAGS = {"x": 11, "dy": 12, "w_qkv": 21, "w_o": 22, "w_gu": 23, "w_d": 24, "g1": 25, "g2": 26}


def _gen(seed, tag, layer, device):
    g = torch.Generator(device=device)
    g.manual_seed((int(seed) * 1000003 + _TAGS[tag] * 7919 + int(layer)) & ((1 << 63) - 1))
    return g


def weight_shapes(cfg):
    d, H, Hkv, Dh, F = cfg["d"], cfg["H"], cfg["Hkv"], cfg["Dh"], cfg["F"]
    return {
        "w_qkv": ((H + 2 * Hkv) * Dh, d),
        "w_o": (d, H * Dh),
        "w_gu": ((F if cfg.get("act") == "relu2" else 2 * F), d),  # [gate; up] or up alone
        "w_d": (d, F),
        "g1": (d,),
        "g2": (d,),
    }


def layer_weights(cfg, layer, seed=0, device="cpu", dtype=torch.bfloat16, std=0.02, gamma_noise=0.0):
    """Weights of one layer: dict name -> tensor ([out, in] row-major)."""
    out = {}
    for name, shape in weight_shapes(cfg).items():
        g = _gen(seed, name, layer, device)
        if name in ("g1", "g2"):
            t = torch.ones(shape, device=device, dtype=torch.float32)
            if gamma_noise:
                t += gamma_noise * torch.randn(shape, generator=g, device=device, dtype=torch.float32)
        else:
            sd = std
            if cfg.get("init") == "depth_scaled" and name in ("w_o", "w_d"):
                sd = std / (2.0 * cfg["L"]) ** 0.5
            t = sd * torch.randn(shape, generator=g, device=device, dtype=torch.float32)
        out[name] = t.to(torch.bfloat16).to(dtype)
    return out


def stack_weights(cfg, seed=0, device="cpu", dtype=torch.bfloat16, std=0.02, gamma_noise=0.0):
    return [layer_weights(cfg, l, seed, device, dtype, std, gamma_noise) for l in range(cfg["L"])]


def activations(cfg, seed=0, device="cpu", dtype=torch.bfloat16, B=None, S=None):
    """x [B, S, d] ~ N(0, 1), bf16-representable."""
    B = cfg["B"] if B is None else B
    S = cfg["S"] if S is None else S
    g = _gen(seed, "x", 0, device)
    t = torch.randn((B, S, cfg["d"]), generator=g, device=device, dtype=torch.float32)
    return t.to(torch.bfloat16).to(dtype)


def upstream_grad(cfg, seed=2, device="cpu", dtype=torch.bfloat16, B=None, S=None):
    """dY [B, S, d] ~ N(0, 1), bf16-representable."""
    B = cfg["B"] if B is None else B
    S = cfg["S"] if S is None else S
    g = _gen(seed, "dy", 0, device)
    t = torch.randn((B, S, cfg["d"]), generator=g, device=device, dtype=torch.float32)
    return t.to(torch.bfloat16).to(dtype)
