"""Host-side pieces of bench.py that need no GPU: the clock-sample summary that
decides whether a run was throttled, and the peak table it reports against."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _sampler(lines):
    c = bench.ClockSampler(0)
    c.out = "\n".join(lines)
    return c.summary()


def test_clock_summary_median_and_reasons():
    rows = [
        "0, 1500, 2070, 1350.1, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
        "0, 1400, 2070, 1398.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
        "0, 1450, 2070, 1380.5, 0x0000000000000000, Not Active, Not Active, Not Active, "
        "Not Active",
    ]
    s = _sampler(rows)
    assert s["sm_mhz"] == 1450 and s["sm_max_mhz"] == 2070 and s["samples"] == 3
    assert s["reasons"] == ["sw_power_cap"]


def test_clock_summary_reports_thermal_and_skips_garbage():
    rows = ["garbage line", "0, [N/A], 2070, 1, x, a, b, c, d",
            "0, 1200, 2070, 900, 0x60, Active, Not Active, Active, Not Active"]
    s = _sampler(rows)
    assert s["samples"] == 1 and s["sm_mhz"] == 1200
    assert s["reasons"] == ["hw_slowdown", "sw_thermal_slowdown"]


def test_clock_summary_without_samples():
    s = _sampler([])
    assert s["sm_mhz"] is None and s["reasons"] == ["unsampled"]


def test_peaks_are_the_measured_file_when_present():
    peaks, src = bench._peaks()
    if os.path.exists(os.path.join(ROOT, "MEASURED_PEAKS.json")):
        assert src == "measured" and peaks["hbm_gbs"] > 1000
    else:
        assert src == "fallback" and peaks["hbm_gbs"] == 6800.0
    assert peaks["bf16_tflops_sustained"] <= peaks["bf16_tflops"]


def test_both_arms_name_the_same_config():
    """The GPU line and the reference line take their config from one function:
    the workload, the whole job's batch and the partition at each N."""
    c1, c8 = bench._config(1), bench._config(8)
    assert c1["global_batch"] == 1024 and c8["global_batch"] == 8 * 1024
    assert c1["workload"] == c8["workload"] and c1["workload"].startswith("moe:")
    assert c1["parallelism"].startswith("dp1") and c8["parallelism"].startswith("dp8")


def test_oracle_sample_step_on_the_tiny_pool():
    """The reference arm's step (full admission + a row sample) runs on the host alone."""
    ref = bench.OracleSampleStep("tiny", 8)
    t, M = ref.run(0, 2)
    assert t > 0 and M == ref.M and 8 <= M <= int(ref.rows.mask.sum())
