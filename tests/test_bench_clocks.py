"""The benchmark's clock record, parsed from nvidia-smi's CSV samples (no GPU: the samples are
written by the test).  A timed region is rejected when it saw a slowdown reason, so the
parser must report every active reason and the median clocks."""
import os
import sys
import tempfile

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


class _Stopped:
    """Stands in for the nvidia-smi process: already finished."""

    def terminate(self):
        pass

    def wait(self, timeout=None):
        return 0


def _sampler(lines):
    fd, path = tempfile.mkstemp(suffix=".csv")
    with os.fdopen(fd, "w") as f:
        f.write("\n".join(lines) + "\n")
    c = bench.ClockSampler(0)
    c.proc, c.path = _Stopped(), path
    return c


def test_medians_reasons_memory_clock_and_temperature():
    lines = [
        "0, 2070, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active, 3996, 55",
        "0, 1980, 2070, 1390.0, 0x4, Not Active, Not Active, Not Active, Active, 3996, 58",
        "0, 2070, 2070, 1200.5, 0x0, Not Active, Not Active, Not Active, Not Active, 3996, 57",
        "garbage line",
    ]
    out = _sampler(lines).stop()
    assert out["sm_mhz"] == 2070.0 and out["sm_max_mhz"] == 2070.0 and out["samples"] == 3
    assert out["reasons"] == ["sw_power_cap"]
    assert out["mem_mhz"] == 3996.0 and out["gpu_temp_c"] == 57.0


def test_slowdown_reasons_are_all_reported_and_old_format_still_parses():
    lines = [
        "0, 1500, 2070, 700.0, 0x8, Active, Not Active, Not Active, Not Active",
        "0, 1400, 2070, 700.0, 0x28, Not Active, Active, Active, Not Active",
    ]
    out = _sampler(lines).stop()
    assert out["reasons"] == ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"]
    assert out["sm_mhz"] == 1450.0
    assert "mem_mhz" not in out
