"""CPU tests of the C ABI: the library loads and exports every function that
include/ld.h declares, argument/shape validation happens on the host, and
the host-side schedule (rates, thresholds, scales) equals the oracle's bit
for bit.  No kernel is launched."""

import ctypes
import os

import pytest

import paper_2609_05275_gb300 as P
from paper_2609_05275_gb300 import synth
from parity import oracle_sched
from oracle import schedule as OS

pytestmark = pytest.mark.skipif(not os.path.exists(P.LIB_PATH), reason="libld.so not built")


def test_exports_every_header_function():
    names = P.header_functions()
    assert {"ld_create", "ld_workspace_size", "ld_set_schedule", "ld_forward", "ld_backward", "ld_destroy",
            "ld_get_masks", "ld_draw_masks", "ld_sync", "ld_status_str", "ld_get_rates", "ld_gemm_bf16"} <= set(names)
    L = P.lib()
    for n in names:
        assert hasattr(L, n), n
    assert P.ld_status_str(P.LD_OK) == "ok"
    assert "timed out" in P.ld_status_str(P.LD_ERR_TIMEOUT)


@pytest.mark.parametrize("name", sorted(synth.CONFIGS))
def test_configs_accepted(name):
    cfg = synth.CONFIGS[name]
    for fp32 in (0, 1):
        assert P.ld_create_status(P.make_config(cfg, fp32_debug=fp32)) == P.LD_OK


@pytest.mark.parametrize("change,status", [
    (dict(Dh=48), P.LD_ERR_SHAPE), (dict(H=6, Hkv=4), P.LD_ERR_SHAPE), (dict(S=100), P.LD_ERR_SHAPE),
    (dict(S=0), P.LD_ERR_SHAPE), (dict(d=100), P.LD_ERR_SHAPE), (dict(F=30), P.LD_ERR_SHAPE),
    (dict(L=0), P.LD_ERR_SHAPE), (dict(B=0), P.LD_ERR_SHAPE), (dict(eps=float("nan")), P.LD_ERR_ARG),
    (dict(alpha=float("inf")), P.LD_ERR_ARG), (dict(rope_theta=-1.0), P.LD_ERR_ARG),
])
def test_create_rejects(change, status):
    cfg = dict(synth.CONFIGS["tiny"], **change)
    assert P.ld_create_status(P.make_config(cfg)) == status


def test_sublayer_flag():
    cfg = synth.CONFIGS["tiny"]
    bad = P.make_config(cfg)
    bad.sublayer = 2
    assert P.ld_create_status(bad) == P.LD_ERR_ARG
    h1, h2 = P.ld_create(P.make_config(cfg)), P.ld_create(P.make_config(cfg, sublayer=True))
    try:
        # the attention and FFN mask tables take twice the mask space, nothing else changes
        n1, n2 = P.ld_workspace_size(h1), P.ld_workspace_size(h2)
        assert n1 <= n2 <= n1 + 3 * 256 + cfg["L"] * cfg["B"] * 5 + cfg["L"] * 4
    finally:
        P.ld_destroy(h1)
        P.ld_destroy(h2)


def test_position_and_activation_flags():
    cfg = synth.CONFIGS["tiny"]
    assert P.ld_create_status(P.make_config(dict(cfg, alibi=True))) == P.LD_ERR_ARG  # ALiBi and RoPE together
    assert P.ld_create_status(P.make_config(dict(cfg, alibi=True, rope_theta=0.0, act="relu2"))) == P.LD_OK
    bad = P.make_config(cfg)
    bad.act = 2
    assert P.ld_create_status(bad) == P.LD_ERR_ARG
    # the squared-ReLU stack saves u instead of g || u: a smaller workspace
    h1 = P.ld_create(P.make_config(cfg))
    h2 = P.ld_create(P.make_config(dict(cfg, rope_theta=0.0, alibi=True, act="relu2")))
    try:
        assert P.ld_workspace_size(h2) < P.ld_workspace_size(h1)
    finally:
        P.ld_destroy(h1)
        P.ld_destroy(h2)


def test_per_token_flag():
    # per-token granularity: no ALiBi; on the bf16 path head size 64 or 128
    # and S % 128 == 0 (the tcgen05 attention), any supported shape on the
    # float32 debug path; the mask tables grow to one entry per token
    cfg = dict(synth.CONFIGS["tiny"])          # Dh = 32, S = 64
    assert P.ld_create_status(P.make_config(cfg, "per_token")) == P.LD_ERR_SHAPE
    assert P.ld_create_status(P.make_config(cfg, "per_token", fp32_debug=True)) == P.LD_OK
    c128 = dict(cfg, H=2, Hkv=1, Dh=128, S=128)
    assert P.ld_create_status(P.make_config(c128, "per_token")) == P.LD_OK
    assert P.ld_create_status(P.make_config(dict(c128, S=192), "per_token")) == P.LD_ERR_SHAPE
    assert P.ld_create_status(P.make_config(dict(c128, H=4, Hkv=2, Dh=64), "per_token")) == P.LD_OK
    assert P.ld_create_status(P.make_config(dict(c128, H=4, Hkv=2, Dh=64, S=192), "per_token")) == P.LD_ERR_SHAPE
    assert P.ld_create_status(P.make_config(dict(c128, alibi=True, rope_theta=0.0), "per_token")) == P.LD_ERR_ARG
    assert P.ld_create_status(P.make_config(dict(c128, alibi=True, rope_theta=0.0), "per_token",
                                            fp32_debug=True)) == P.LD_ERR_ARG
    bad = P.make_config(c128)
    bad.granularity = 4
    assert P.ld_create_status(bad) == P.LD_ERR_ARG
    h1, h2 = P.ld_create(P.make_config(c128)), P.ld_create(P.make_config(c128, "per_token"))
    try:
        n1, n2 = P.ld_workspace_size(h1), P.ld_workspace_size(h2)
        # at least (S - 1) more mask bytes and (S - 1) more kept-list ints per (layer, sequence)
        assert n2 - n1 >= c128["L"] * c128["B"] * (c128["S"] - 1) * 5 - 4096
    finally:
        P.ld_destroy(h1)
        P.ld_destroy(h2)


def test_eval_entry_points():
    cfg = synth.CONFIGS["llama8b"]
    h = P.ld_create(P.make_config(cfg))
    try:
        # one layer's activations instead of L layers' plus the backward scratch
        assert P.ld_eval_workspace_size(h) * 8 < P.ld_workspace_size(h)
        L = P.lib()
        W = (P.ld_layer_w * cfg["L"])()
        ex = (ctypes.c_ubyte * cfg["L"])(*([1] + [0] * (cfg["L"] - 1)))
        fake = ctypes.c_void_p(1 << 20)  # aligned, never dereferenced: argument checks fail first
        assert L.ld_forward_eval(h, ex, None, W, fake, fake, None) == P.LD_ERR_ARG  # layer 0's weights missing
        ex2 = (ctypes.c_ubyte * cfg["L"])(*([2] + [0] * (cfg["L"] - 1)))
        assert L.ld_forward_eval(h, ex2, None, W, fake, fake, None) == P.LD_ERR_ARG  # not 0/1
        assert L.ld_forward_eval(h, None, None, W, fake, fake, None) == P.LD_ERR_ARG
        zero = (ctypes.c_ubyte * cfg["L"])()
        rv = (ctypes.c_float * cfg["L"])(*([float("nan")] * cfg["L"]))
        assert L.ld_forward_eval(h, zero, rv, W, fake, fake, None) == P.LD_ERR_ARG  # non-finite r_eval
    finally:
        P.ld_destroy(h)


def test_schedule_validation_and_state():
    h = P.ld_create(P.make_config(synth.CONFIGS["tiny"]))
    try:
        L = P.lib()
        # rates before a schedule: state error
        p = (ctypes.c_double * 2)()
        assert L.ld_get_rates(h, 0, p, None, None) == P.LD_ERR_STATE
        bad = [dict(dist="uniform", p_max=1.5), dict(dist="uniform", p_max=float("nan")),
               dict(dist="explicit", p_explicit=[0.0, -0.1]), dict(dist="ild", p_max=0.2, time="its", T=1),
               dict(dist="ild", p_max=0.2, time="ramp", ramp=(10, 10, 0.0, 1.0))]
        for s in bad:
            assert P.ld_set_schedule_status(h, P.make_schedule(s)) == P.LD_ERR_ARG, s
        # backward without forward: argument errors first, then a state error
        # (the pointers below are aligned and never dereferenced: the checks
        # run on the host before any device work)
        assert L.ld_backward(h, None, None, None, None, None) == P.LD_ERR_ARG
        cfg = synth.CONFIGS["tiny"]
        fake = ctypes.c_void_p(1 << 20)
        W = (P.ld_layer_w * cfg["L"])(*[P.ld_layer_w(*([1 << 20] * 6)) for _ in range(cfg["L"])])
        G = (P.ld_layer_g * cfg["L"])(*[P.ld_layer_g(*([1 << 20] * 6)) for _ in range(cfg["L"])])
        assert L.ld_backward(h, W, fake, G, fake, None) == P.LD_ERR_STATE
        Wmis = (P.ld_layer_w * cfg["L"])(*[P.ld_layer_w(*([(1 << 20) + 4] * 6)) for _ in range(cfg["L"])])
        assert L.ld_backward(h, Wmis, fake, G, fake, None) == P.LD_ERR_ARG  # misaligned weights
        assert L.ld_get_masks(h, None, None, None) == P.LD_ERR_STATE
        assert L.ld_create(None, None) == P.LD_ERR_ARG
    finally:
        P.ld_destroy(h)


SCHEDS = [
    dict(dist="ild", p_max=0.4, time="const"),
    dict(dist="uniform", p_max=0.3, time="its", T=1000),
    dict(dist="ild", p_max=0.99, time="dts", T=777),
    dict(dist="ald", p_max=0.2, time="const"),
    dict(dist="ild", p_max=0.3, time="ramp", ramp=(0, 1000, 0.0, 1.0)),
    dict(dist="explicit", p_explicit=[0.0, 0.5, 1.0, 0.125, 0.3, 0.7], time="const"),
]


@pytest.mark.parametrize("sched", SCHEDS, ids=lambda s: f"{s['dist']}-{s.get('time')}")
@pytest.mark.parametrize("L", [1, 6, 13, 32])
def test_rates_match_oracle_bit_exact(sched, L):
    if sched["dist"] == "explicit":
        sched = dict(sched, p_explicit=(sched["p_explicit"] * 6)[:L])
    cfg = dict(synth.CONFIGS["tiny"], L=L)
    h = P.ld_create(P.make_config(cfg))
    try:
        P.ld_set_schedule(h, P.make_schedule(dict(sched, seed=3)))
        for t in (0, 1, 250, 500, 776, 999, 2000):
            p, thr, sc = P.ld_get_rates(h, t, L)
            ref = OS.layer_rates(oracle_sched(sched), L, t)
            assert p == ref
            assert thr == [OS.drop_threshold(v) for v in ref]
            for a, v in zip(sc, ref):
                r = OS.residual_scale(v, 1.0)
                assert abs(a - r) <= 1e-7 * max(1.0, r)
    finally:
        P.ld_destroy(h)


def test_workspace_grows_with_batch():
    c1 = synth.CONFIGS["gpt2"]
    c2 = dict(c1, B=2 * c1["B"])
    h1, h2 = P.ld_create(P.make_config(c1)), P.ld_create(P.make_config(c2))
    try:
        assert P.ld_workspace_size(h2) > 1.9 * P.ld_workspace_size(h1)
    finally:
        P.ld_destroy(h1)
        P.ld_destroy(h2)
