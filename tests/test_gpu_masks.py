"""Masks and kept-sequence (per token: kept-token) lists of the device kernel
against the oracle, bit for bit: every workload schedule at its benchmark
steps, and the whole drop-rate / distribution / granularity / seed sweep on
the 1.3B shape."""

import numpy as np
import pytest
import torch

import paper_2609_05275_gb300 as P
from paper_2609_05275_gb300 import synth
from parity import oracle_masks, oracle_sched
from oracle import masks as OM
from oracle import schedule as OS

pytestmark = pytest.mark.gpu


def _check(cfg, sched, steps, granularity, sublayer=False):
    st = P.LayerDropStack(cfg, sched, granularity=granularity, sublayer=sublayer)
    try:
        for t in steps:
            mask, idx, cnt = st.draw_masks(t)
            ref, _, _ = oracle_masks(cfg, sched, t, granularity, sublayer)
            if granularity == "per_token":
                ridx, rcnt, _ = OM.kept_token_lists(ref)
            else:
                ridx, rcnt = OM.kept_lists(ref)
            assert (mask == ref).all(), t
            assert (cnt == rcnt).all(), t
            assert (idx == ridx).all(), t
    finally:
        st.close()


@pytest.mark.parametrize("name", sorted(synth.CONFIGS))
@pytest.mark.parametrize("granularity", ["per_sequence", "per_batch"])
def test_workload_masks(name, granularity):
    cfg = synth.CONFIGS[name]
    _check(cfg, synth.SCHEDULES[name], synth.STEPS[name] + [1, 2 ** 33 + 17], granularity)


def test_sweep_masks():
    sw = synth.SWEEP
    cfg = synth.CONFIGS[sw["base"]]
    for p_max in sw["p_max"]:
        for dist in sw["dist"]:
            for gran in sw["granularity"]:
                for seed in (sw["seeds"][0], sw["seeds"][7], sw["seeds"][-1]):
                    _check(cfg, dict(dist=dist, p_max=p_max, time="const", seed=seed), [0], gran)
    # all 20 seeds of one cell
    for seed in sw["seeds"]:
        _check(cfg, dict(dist="ild", p_max=0.5, time="const", seed=seed), [0], "per_sequence")


@pytest.mark.parametrize("B", [1, 31, 32, 33, 1000, 4096])
def test_large_and_ragged_batches(B):
    cfg = dict(synth.CONFIGS["tiny"], B=B, L=5)
    sched = dict(dist="explicit", p_explicit=[0.0, 1.0, 0.5, 0.1, 0.9], time="const", seed=2 ** 40 + 3)
    _check(cfg, sched, [0, 7], "per_sequence")


@pytest.mark.parametrize("granularity", ["per_sequence", "per_batch"])
@pytest.mark.parametrize("B", [4, 33, 4096])
def test_sublayer_masks(granularity, B):
    # attention (word 0) and FFN (word 1) tables, bit for bit
    cfg = dict(synth.CONFIGS["tiny"], B=B, L=7)
    sched = dict(dist="ild", p_max=0.8, time="const", seed=2 ** 35 + 9)
    _check(cfg, sched, [0, 5, 2 ** 33 + 1], granularity, sublayer=True)


@pytest.mark.parametrize("b_offset", [0, 8, 1000])
def test_per_shard_masks(b_offset):
    # per-device batch dropping: one draw per layer and step for the shard,
    # keyed by its first global sequence; bit-exact against the oracle
    cfg = dict(synth.CONFIGS["tiny"], B=8, L=6)
    sched = dict(dist="ild", p_max=0.7, time="const", seed=77)
    st = P.LayerDropStack(cfg, sched, granularity="per_shard", b_offset=b_offset)
    try:
        rates = OS.layer_rates(oracle_sched(sched), cfg["L"], 3)
        thr = [OS.drop_threshold(p) for p in rates]
        mask, idx, cnt = st.draw_masks(3)
        ref = OM.draw_masks(77, 3, thr, cfg["B"], OM.PER_SHARD, b_offset=b_offset)
        ridx, rcnt = OM.kept_lists(ref)
        assert (mask == ref).all() and (idx == ridx).all() and (cnt == rcnt).all()
        assert ((cnt == 0) | (cnt == cfg["B"])).all()  # whole shard kept or dropped
    finally:
        st.close()
