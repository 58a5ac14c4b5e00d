"""Per-layer, per-step drop rates p^{l,t} and the derived per-layer constants.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

Follows:
  * Dropout Distribution section: uniform p = p_max; increasing layer
    distribution (ILD) p = l/(L-1) * p_max; alternating layer distribution
    (ALD) p = p_max * 1[l odd], l = 0..L-1.
  * Dropout Schedule section: constant; increasing time schedule (ITS)
    p = p_dist * t/(T-1); decreasing time schedule (DTS)
    p = p_dist * (1 - t/(T-1)).  The body uses T-1; the glossary prints t/T.
    T-1 is used here because it is the reading under which the paper's
    closed form for the mean rate (0.25 p_max for ILD+DTS) is exact.
  * Dropout Scale paragraph: r_train = 1/rho with rho = 1 - p; the
    parameterization table multiplies the residual branch by m_L^{-1} rho^{-1},
    which is alpha * (1/rho) here with alpha = m_L^{-1} (default 1).
  * A linear warm-up ramp of the rate (not in the paper) is provided as a
    fourth time schedule: factor s0 + (s1 - s0) * clamp((t-t0)/(t1-t0), 0, 1).

All arithmetic is in Python floats (IEEE binary64), in the order written
below; float32 inputs are widened exactly before use.
"""

import math

import numpy as np

# Layer distributions and time schedules (own numbering of the oracle).
UNIFORM, ILD, ALD, EXPLICIT = "uniform", "ild", "ald", "explicit"
CONST, ITS, DTS, RAMP = "const", "its", "dts", "ramp"

TWO32 = 4294967296.0


def f32(v):
    """Widen a value that the schedule stores as float32 to binary64 exactly."""
    return float(np.float32(v))


def dist_rate(dist, p_max, layer, L, p_explicit=None):
    """p^l_dist of the Dropout Distribution section (before the time factor)."""
    p_max = f32(p_max)
    if dist == UNIFORM:
        return p_max
    if dist == ILD:
        if L == 1:
            # l/(L-1) is undefined for one layer; the distribution "starts at
            # 0 at the first layer", so the only layer gets rate 0.
            return 0.0
        return (p_max * layer) / (L - 1)
    if dist == ALD:
        return p_max if layer % 2 == 1 else 0.0
    if dist == EXPLICIT:
        return f32(p_explicit[layer])
    raise ValueError(f"unknown distribution {dist!r}")


def time_factor(kind, t, T=None, ramp=None):
    """Multiplier of p^l_dist at step t (Dropout Schedule section)."""
    if kind == CONST:
        return 1.0
    if kind == ITS:
        return t / (T - 1)
    if kind == DTS:
        return 1.0 - t / (T - 1)
    if kind == RAMP:
        t0, t1, s0, s1 = ramp
        s0, s1 = f32(s0), f32(s1)
        frac = (t - t0) / (t1 - t0)
        frac = min(max(frac, 0.0), 1.0)
        return s0 + (s1 - s0) * frac
    raise ValueError(f"unknown time schedule {kind!r}")


def layer_rates(sched, L, t):
    """p^{l,t} for l = 0..L-1: distribution times time factor, clamped to [0,1].

    ``sched`` is a dict with keys dist, p_max, p_explicit (optional),
    time, T, ramp=(t0, t1, s0, s1).
    """
    out = []
    for layer in range(L):
        d = dist_rate(sched["dist"], sched.get("p_max", 0.0), layer, L, sched.get("p_explicit"))
        tf = time_factor(sched.get("time", CONST), t, sched.get("T"), sched.get("ramp"))
        p = d * tf
        p = min(max(p, 0.0), 1.0)
        out.append(p)
    return out


def drop_threshold(p):
    """Integer threshold on a uniform 32-bit word: the layer is dropped for a
    sequence iff its word u < thr.  thr = floor(p * 2^32), so P(drop) is p to
    within 2^-32, p = 0 never drops and p = 1 always drops."""
    return int(math.floor(p * TWO32))


def residual_scale(p, alpha=1.0):
    """r_train * m_L^{-1} = alpha / (1 - p), the factor on both residual
    branches of a kept layer.  p = 1 keeps no row, so the factor is never
    used; it is defined as 0 there."""
    if p >= 1.0:
        return 0.0
    return f32(alpha) / (1.0 - p)


def p_mean(rates):
    """p^t_mean = (1/L) sum_l p^{l,t}, the FLOPs saving at step t."""
    return sum(rates) / len(rates)


def p_bar(sched, L, T):
    """P-bar = (1/T) sum_t (1/L) sum_l p^{l,t}: the total FLOPs saving."""
    return sum(p_mean(layer_rates(sched, L, t)) for t in range(T)) / T


def effective_depth(rates):
    """Expected number of layers a sequence executes: sum_l (1 - p_l)."""
    return sum(1.0 - p for p in rates)
