"""Host logic of bench.py, on the CPU: the clock summary it adds to every line (median SM
clock, throttle reasons decoded from NVML's bit mask), the measured peak it divides by, and
the scaling of the committed DRAM-traffic record to a launch."""
import json
import os

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    import bench as b

    return b


def test_clock_summary_median_and_reasons(bench):
    s = bench.ClockSampler(None)
    s.max_mhz = 2070
    # (SM MHz, reason bits): idle (0x1) is not a reason; sw_power_cap 0x4, hw_slowdown 0x8
    s.samples = [(2070, 0x1), (1980, 0x4), (2010, 0x0), (1500, 0x4 | 0x8), (2070, 0x0)]
    out = s.summary()
    assert out["sm_mhz"] == 2010 and out["sm_max_mhz"] == 2070 and out["samples"] == 5
    assert out["reasons"] == ["hw_slowdown", "sw_power_cap"]


def test_clock_summary_without_samples(bench):
    s = bench.ClockSampler(None)
    s.samples = []
    out = s.summary()
    assert out["sm_mhz"] is None and out["reasons"] == [] and out["samples"] == 0


def test_peak_is_the_measured_copy_bandwidth(bench):
    with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
        want = float(json.load(f)["hbm_gbs"])
    assert bench.hbm_peak() == (want, "measured")


def test_traffic_record_scales_with_algorithmic_bytes(bench, monkeypatch):
    """A record applies only to the kernel source it was taken on (its hash), and then scales
    by algorithmic bytes; the source hash is pinned here so the test checks the logic alone."""
    with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
        rec = json.load(f)["workloads"]
    for key, e in rec.items():
        monkeypatch.setattr(bench, "kernel_source_sha", lambda: e["kernel_source_sha"])
        got = bench.recorded_traffic(key, 2.0 * e["algorithmic_bytes_per_launch"])
        assert got == pytest.approx(2.0 * e["dram_bytes_per_launch"])
        monkeypatch.setattr(bench, "kernel_source_sha", lambda: "another source")
        assert bench.recorded_traffic(key, 1e9) is None
    assert bench.recorded_traffic("no_such_workload", 1e9) is None


def test_forward_kernel_label(bench, monkeypatch):
    """The forward line names the kernel that runs: the paired-item kernel where pbb_forward
    takes two query tiles per CTA, else the one-item kernel with its CTAs per SM."""
    import paper_2606_02680_gb300 as pbb
    from paper_2606_02680_gb300 import inputs

    w = inputs.FORWARD_WORKLOADS["fwd_b2_n32768_B4096"]
    monkeypatch.setattr(pbb, "plan_forward", lambda *a: (128, 1))
    monkeypatch.setattr(pbb, "plan_forward_query_tiles", lambda *a: 2)
    assert bench.fwd_kernel_label(w) == "forward_pair_kernel<128,4,128 keys,2 query tiles per CTA>"
    monkeypatch.setattr(pbb, "plan_forward", lambda *a: (32, 3))
    monkeypatch.setattr(pbb, "plan_forward_query_tiles", lambda *a: 1)
    w = inputs.FORWARD_WORKLOADS["fwd_b16_n8192_B128"]
    assert bench.fwd_kernel_label(w) == "forward_kernel<64,4,32 keys,3 CTAs/SM>"
