"""Host logic of bench.py that needs no GPU: the clock/throttle record, the
roofline's recorded DRAM traffic and its source-hash guard, the peak
denominators and the algorithmic byte count of one step."""
import json

import pytest

import bench
from paper_2607_09694_gb300 import sites


class _FakeProc:
    def terminate(self):
        pass

    def wait(self, timeout=None):
        return 0


def _sampler(lines):
    s = bench.ClockSampler(0)
    s.proc = _FakeProc()
    s.lines = list(lines)
    return s


def test_clock_record_median_max_and_reasons():
    lines = [
        "0, 2070, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active",
        "0, 2055, 2070, 1350.0, 0x4, Not Active, Not Active, Not Active, Active",
        "0, 1980, 2070, 1399.5, 0x8, Active, Not Active, Not Active, Not Active",
        "garbage line",
        "0, [N/A], 2070, 10, 0x0, Not Active, Not Active, Not Active, Not Active",
    ]
    rec = _sampler(lines).stop()
    assert rec["sm_mhz"] == 2055.0 and rec["sm_max_mhz"] == 2070.0 and rec["samples"] == 3
    assert rec["reasons"] == ["hw_slowdown", "sw_power_cap"]


def test_clock_record_without_nvidia_smi():
    s = bench.ClockSampler(0)
    assert s.stop()["reasons"] == ["nvidia-smi unavailable"]


def test_recorded_traffic_follows_the_source_hash(tmp_path, monkeypatch):
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "k_traffic.txt").write_text(
        "# comment: with a colon\nsource_hash: abc123\ndram_bytes_per_launch_avg: 2588475021\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setattr(bench, "_kernel_source_hash", lambda: "abc123")
    assert bench._recorded_traffic("k") == 2588475021.0
    monkeypatch.setattr(bench, "_kernel_source_hash", lambda: "changed")
    assert bench._recorded_traffic("k") is None  # counters taken on other sources are not reported
    assert bench._recorded_traffic("missing") is None


def test_peaks_measured_or_fallback(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench._peaks() == (bench.FALLBACK_HBM_GBS, "fallback")
    (tmp_path / "MEASURED_PEAKS.json").write_text(json.dumps({"hbm_gbs": 6682.5, "bf16_tflops": 1965.9}))
    assert bench._peaks() == (6682.5, "measured")
    assert bench._bf16_peak() == (1965.9, "measured")


def test_step_bytes_match_the_per_site_counts():
    """One step: 49 forwards and 49 backwards, the first backward (site 49)
    writing the gradients and the others accumulating.  The headline site
    (n = 49, T = 16384, d = 1024, bf16) moves F = 1.678 GB forward and
    B = 3.322 GB backward with the gradients written, 4.966 GB accumulated."""
    fwd, bwd = bench.site_bytes()
    assert len(fwd) == len(bwd) == 49
    assert fwd[48] == pytest.approx(1.678e9, rel=1e-3)
    assert bwd[48] == pytest.approx(3.322e9, rel=1e-3)
    acc49 = sites.backward_bytes(sites.SiteShape("sliced", 49, 16384, 1024, 16, accumulate=1))
    assert acc49 == pytest.approx(4.966e9, rel=1e-3)
    assert sum(fwd) + sum(bwd) == 166067306496
    # a site's bytes grow linearly with its sources
    assert all(fwd[t + 1] - fwd[t] == fwd[1] - fwd[0] for t in range(47))
