"""Pins of the oracle's schedule arithmetic against what the paper fixes:
the closed forms of the Dropout Distribution / Dropout Schedule sections and
the effective-depth footnote, and the FLOPs savings printed in its tables
(fixture tests/golden/flops_savings.txt)."""

import math
import os

import pytest

from oracle import schedule as S

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "flops_savings.txt")


def _sched(dist, p_max, time="const", T=None, ramp=None):
    return dict(dist=dist, p_max=p_max, time=time, T=T, ramp=ramp)


@pytest.mark.parametrize("L", [2, 3, 12, 13, 24, 32, 52])
def test_ild_mean_is_half_pmax(L):
    # Dropout Distribution section: p_mean(ILD) = 0.5 p_max (arithmetic series).
    for p_max in (0.1, 0.25, 0.4, 0.99):
        rates = S.layer_rates(_sched("ild", p_max), L, 0)
        assert rates[0] == 0.0
        assert rates[-1] == pytest.approx(S.f32(p_max), abs=1e-15)
        assert S.p_mean(rates) == pytest.approx(0.5 * S.f32(p_max), abs=1e-12)


@pytest.mark.parametrize("L", [2, 3, 12, 13, 17, 23, 32])
def test_ald_mean_closed_form(L):
    # p_mean(ALD) = floor(L/2)/L * p_max; layer 0 (even) is never dropped.
    p_max = 0.4
    rates = S.layer_rates(_sched("ald", p_max), L, 0)
    assert rates[0] == 0.0
    assert all(rates[l] == (S.f32(p_max) if l % 2 else 0.0) for l in range(L))
    assert S.p_mean(rates) == pytest.approx((L // 2) / L * S.f32(p_max), abs=1e-12)


def test_ald_13_layers_is_not_exactly_ten_percent():
    # The distribution table labels ALD p_max 0.2 at L = 13 as "10%"; the exact
    # value of the definition is 6/13 * 0.2.
    v = S.p_mean(S.layer_rates(_sched("ald", 0.2), 13, 0))
    assert v == pytest.approx(6 / 13 * S.f32(0.2), abs=1e-12)
    assert abs(v - 0.10) > 0.005


@pytest.mark.parametrize("T", [2, 5, 100, 1001])
@pytest.mark.parametrize("L", [2, 13, 32])
def test_pbar_closed_forms(L, T):
    # Dropout Schedule section: P-bar(uniform, ITS) = 0.5 p_max and
    # P-bar(ILD, ITS) = P-bar(ILD, DTS) = 0.25 p_max.
    p = 0.8
    pm = S.f32(p)
    assert S.p_bar(_sched("uniform", p, "its", T), L, T) == pytest.approx(0.5 * pm, abs=1e-12)
    assert S.p_bar(_sched("ild", p, "its", T), L, T) == pytest.approx(0.25 * pm, abs=1e-12)
    assert S.p_bar(_sched("ild", p, "dts", T), L, T) == pytest.approx(0.25 * pm, abs=1e-12)
    assert S.p_bar(_sched("uniform", p, "dts", T), L, T) == pytest.approx(0.5 * pm, abs=1e-12)
    assert S.p_bar(_sched("ild", p, "const", T), L, T) == pytest.approx(0.5 * pm, abs=1e-12)


def test_schedule_endpoints():
    # ITS starts at 0 and reaches p_dist at t = T-1; DTS the reverse.
    T, L = 50, 8
    its0 = S.layer_rates(_sched("uniform", 0.3, "its", T), L, 0)
    its1 = S.layer_rates(_sched("uniform", 0.3, "its", T), L, T - 1)
    dts0 = S.layer_rates(_sched("uniform", 0.3, "dts", T), L, 0)
    dts1 = S.layer_rates(_sched("uniform", 0.3, "dts", T), L, T - 1)
    assert its0 == [0.0] * L and dts1 == [0.0] * L
    assert its1 == dts0 == [S.f32(0.3)] * L


@pytest.mark.parametrize("p_max", [0.2, 0.6, 0.8, 0.99])
@pytest.mark.parametrize("L", [13, 30, 40, 52])
def test_effective_depth(L, p_max):
    # Footnote of the large-scale runs: sum_l (1 - p_max l/(L-1)) = (1 - 0.5 p_max) L.
    rates = S.layer_rates(_sched("ild", p_max), L, 0)
    assert S.effective_depth(rates) == pytest.approx((1 - 0.5 * S.f32(p_max)) * L, abs=1e-10)


def _golden_rows():
    rows = []
    for line in open(GOLDEN):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        table, model, L, p_max, dist, time, printed = line.split()
        rows.append((table, model, int(L), float(p_max), dist, time, float(printed)))
    return rows


@pytest.mark.parametrize("row", _golden_rows(), ids=lambda r: f"{r[0]}-{r[1]}-{r[4]}-{r[5]}-{r[3]}")
def test_printed_flops_savings(row):
    table, model, L, p_max, dist, time, printed = row
    T = 1000
    v = S.p_bar(_sched(dist, p_max, time, T), L, T)
    # The labels are rounded to whole percent (0.2475 -> 25%).  ALD rows carry
    # the label of the group they are compared in: floor(L/2)/L p_max is
    # 0.185 for p_max 0.4 at L = 13, printed in the "20%" group.
    assert abs(v - printed) <= (0.02 if dist == "ald" else 0.01)
    if dist in ("uniform", "ild") or L % 2 == 0:
        # exact for every row whose definition lands on the label
        exact = {"uniform": 1.0, "ild": 0.5, "ald": (L // 2) / L}[dist] * (0.5 if time != "const" else 1.0)
        assert v == pytest.approx(exact * S.f32(p_max), abs=1e-12)
    if table == "hero" and p_max == 0.99:
        assert v == pytest.approx(0.2475, abs=1e-6)


def test_ramp_schedule():
    # Warm-up ramp 0 -> 1 over the first 1000 steps, sampled at 0 / 500 / 2000.
    sch = dict(dist="ild", p_max=0.3, time="ramp", ramp=(0, 1000, 0.0, 1.0))
    for t, f in ((0, 0.0), (500, 0.5), (2000, 1.0)):
        rates = S.layer_rates(sch, 24, t)
        assert rates[-1] == pytest.approx(S.f32(0.3) * f, abs=1e-15)
        assert S.p_mean(rates) == pytest.approx(0.5 * S.f32(0.3) * f, abs=1e-12)


def test_threshold_edges():
    assert S.drop_threshold(0.0) == 0
    assert S.drop_threshold(1.0) == 2 ** 32
    assert S.drop_threshold(0.5) == 2 ** 31
    assert S.drop_threshold(2.0 ** -32) == 1
    assert S.drop_threshold(math.nextafter(1.0, 0.0)) == 2 ** 32 - 1
    assert S.residual_scale(1.0) == 0.0
    assert S.residual_scale(0.0) == 1.0
    assert S.residual_scale(0.5, alpha=0.5) == 1.0


def test_single_layer_ild_and_clamp():
    assert S.layer_rates(_sched("ild", 0.9), 1, 0) == [0.0]
    # p is clamped to [0, 1] (a ramp factor above 1 would overshoot).
    sch = dict(dist="uniform", p_max=0.8, time="ramp", ramp=(0, 10, 0.0, 2.0))
    assert S.layer_rates(sch, 3, 10) == [1.0, 1.0, 1.0]
