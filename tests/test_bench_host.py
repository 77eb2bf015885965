"""Host-side helpers of bench.py (CPU only): the nvidia-smi clock record and the GPU
index it samples."""
import bench


def _sampler(lines):
    c = bench.ClockSampler("0")
    c.lines = lines
    return c.summary()


def test_clock_summary_median_and_reasons():
    lines = ["2070, 2070, 900.1, Not Active, Not Active, Not Active, Active",
             "2062, 2070, 910.0, Not Active, Not Active, Not Active, Not Active",
             "2070, 2070, 905.3, Not Active, Not Active, Not Active, Active"]
    s = _sampler(lines)
    assert s["sm_mhz"] == 2070.0 and s["sm_max_mhz"] == 2070.0 and s["samples"] == 3
    assert s["reasons"] == ["sw_power_cap"]


def test_clock_summary_flags_thermal_and_skips_bad_rows():
    lines = ["garbage", "[N/A], 2070, 1.0, Not Active, Not Active, Not Active, Not Active",
             "1500, 2070, 1300.0, Active, Not Active, Active, Not Active"]
    s = _sampler(lines)
    assert s["samples"] == 1 and s["sm_mhz"] == 1500.0
    assert s["reasons"] == ["hw_slowdown", "sw_thermal_slowdown"]


def test_clock_summary_without_samples():
    s = _sampler([])
    assert s["samples"] == 0 and s["sm_mhz"] is None and s["reasons"] == []


def test_smi_index_follows_visible_devices(monkeypatch):
    monkeypatch.setenv("CUDA_VISIBLE_DEVICES", "3,GPU-abc")
    assert bench.smi_index(0) == "3" and bench.smi_index(1) == "GPU-abc"
    monkeypatch.delenv("CUDA_VISIBLE_DEVICES")
    assert bench.smi_index(2) == "2"
