"""bench.py's clock rule: which clock records rule a timed region's number out (and make it time the steps again)."""
import importlib.util
import os

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_clocks_rejected():
    rej = _bench().clocks_rejected
    full = {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0}
    assert not rej(dict(full, reasons=[]))
    # a power cap under load is normal and kept
    assert not rej(dict(full, reasons=["sw_power_cap"]))
    assert not rej({"sm_mhz": 1500.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"]})
    # any hardware or thermal slowdown rules the number out
    for r in ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"):
        assert rej(dict(full, reasons=[r]))
        assert rej(dict(full, reasons=["sw_power_cap", r]))
    # clocks well below their maximum with no reason: a leftover clock lock
    assert rej({"sm_mhz": 1200.0, "sm_max_mhz": 2070.0, "reasons": []})
    assert not rej({"sm_mhz": 1900.0, "sm_max_mhz": 2070.0, "reasons": []})
    # no record at all is not a reason to time again
    assert not rej({"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]})
    assert not rej({"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]})
