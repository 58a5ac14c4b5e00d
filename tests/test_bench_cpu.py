"""Host logic of bench.py that needs no GPU: the clock-record rule that
rejects a timing (a slowdown, or a clock stuck low with no reason)."""

import bench


def rec(mhz, reasons, mx=2070.0):
    return {"sm_mhz": mhz, "sm_max_mhz": mx, "reasons": reasons, "samples": 10}


def test_power_cap_is_kept():
    assert not bench.clocks_rejected(rec(1672.0, ["sw_power_cap"]))
    assert not bench.clocks_rejected(rec(1200.0, ["sw_power_cap"]))


def test_slowdowns_are_rejected():
    for r in bench.SLOWDOWNS:
        assert bench.clocks_rejected(rec(2000.0, [r]))
        assert bench.clocks_rejected(rec(1600.0, ["sw_power_cap", r]))


def test_stuck_clock_without_reason_is_rejected():
    assert bench.clocks_rejected(rec(1000.0, []))
    assert not bench.clocks_rejected(rec(1900.0, []))


def test_no_record_is_not_rejected():
    assert not bench.clocks_rejected(None)
