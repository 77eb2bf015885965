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


def test_backward_launch_count():
    """Pre, main and post per backward call, except for sequences of at most two key tiles
    at d = 80 / 128, whose main kernel writes dq (no post launch); d = 64 always has three."""
    import bench
    assert bench.bwd_launches(256, 128) == 2 and bench.bwd_launches(130, 80) == 2
    assert bench.bwd_launches(257, 128) == 3 and bench.bwd_launches(8192, 128) == 3
    assert bench.bwd_launches(256, 64) == 3
