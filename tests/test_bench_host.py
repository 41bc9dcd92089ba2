"""Host-side pieces of bench.py that decide what the JSON line reports (no GPU)."""
import datetime
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _line(t, sm, reasons=("Not Active",) * 4):
    ts = datetime.datetime.fromtimestamp(t).strftime("%Y/%m/%d %H:%M:%S.%f")[:-3]
    return ", ".join([ts, "0", str(sm), "2070", "500.0", "90", *reasons])


def test_clock_samples_outside_the_timed_windows_are_ignored():
    t = 1_800_000_000.0
    lines = [_line(t + 0.00, 600), _line(t + 0.02, 2070), _line(t + 0.04, 2055),
             _line(t + 0.06, 2070, ("Not Active", "Not Active", "Not Active", "Active")),
             _line(t + 0.50, 345, ("Active", "Not Active", "Not Active", "Not Active"))]
    got = bench.ClockSampler.parse(lines, [(t + 0.01, t + 0.07)])
    assert got["samples"] == 5 and got["samples_under_load"] == 3
    assert got["sm_mhz"] == 2070 and got["sm_min_mhz"] == 2055 and got["sm_max_mhz"] == 2070
    # hw_slowdown fell outside the windows; sw_power_cap inside
    assert got["reasons"] == ["sw_power_cap"]


def test_clock_parse_without_samples_in_the_windows():
    t = 1_800_000_000.0
    got = bench.ClockSampler.parse([_line(t, 2070), "garbage"], [(t + 5, t + 6)])
    assert got["sm_mhz"] is None and got["samples_under_load"] == 0 and got["samples"] == 1


def test_traffic_vs_dnf_counts_at_least_one_write_of_o():
    # a launch that leaves most of O dirty in L2: reads = inputs, few writes
    dnf, o = 100.0, 25.0
    f = bench.traffic_fields({"read": 75.0, "write": 1.0}, dnf, o)
    assert f["traffic"] == 76.0 and f["dram_read"] == 75.0 and f["dram_write"] == 1.0
    assert f["traffic_vs_dnf"] == 1.0
    f = bench.traffic_fields({"read": 80.0, "write": 30.0}, dnf, o)
    assert f["traffic_vs_dnf"] == 1.1
    assert bench.traffic_fields(None, dnf, o)["traffic"] is None


def test_profile_traffic_needs_the_current_kernel_source(tmp_path, monkeypatch):
    good = tmp_path / "good.txt"
    good.write_text(f"kernel_source_sha256: {bench.kernel_source_hash()}\n"
                    "dram_read_bytes_per_launch: 402890000\ndram_write_bytes_per_launch: 114010000\n")
    stale = tmp_path / "stale.txt"
    stale.write_text("kernel_source_sha256: " + "0" * 64 + "\n"
                     "dram_read_bytes_per_launch: 1\ndram_write_bytes_per_launch: 2\n")
    monkeypatch.setattr(bench, "PROFILES", {3: str(good), 5: str(stale)})
    assert bench.profiled_traffic(3) == {"read": 402890000.0, "write": 114010000.0}
    assert bench.profiled_traffic(5) is None
    assert bench.profiled_traffic(2) is None


def test_default_workload_is_the_largest_single_gpu_case():
    from paper_2606_07713_gb300 import inputs as I
    s = I.CONFIGS[bench.DEFAULT_WORKLOAD].shape
    flops = {cid: 2.0 * c.shape.B * c.shape.H * c.shape.N_q * c.shape.N_k * (c.shape.d_k + c.shape.d_v)
             for cid, c in I.CONFIGS.items()}
    assert max(flops, key=flops.get) == bench.DEFAULT_WORKLOAD
    assert (s.N_q, s.N_k, s.d_k) == (32768, 32768, 128)


def test_job_value_strong_and_weak():
    # strong: the job's FLOPs are fixed; weak (replicas): they grow with the rank count
    assert bench.job_tflops(1e12, 10, 1000.0) == pytest.approx(10.0)
    assert bench.whole_job_tflops(1e12, 10, 4, 1000.0) == pytest.approx(40.0)


def test_rank_slices_weak_and_strong():
    from paper_2606_07713_gb300 import shard as SH
    # weak: rank r owns instance r of the job (its own seed), bh slices each
    for world in (1, 2, 3, 8):
        got = [bench.rank_slices("weak", 16, world, r, 5) for r in range(world)]
        assert [(lo, hi) for lo, hi, _, _ in got] == [(16 * r, 16 * (r + 1)) for r in range(world)]
        assert all(js == 16 * world for _, _, js, _ in got)
        assert [sd for _, _, _, sd in got] == [5 + 1000 * r for r in range(world)]
    # strong: the workload's own slices split; every rank keeps the workload's seed
    got = [bench.rank_slices("strong", 14, 4, r, 3) for r in range(4)]
    assert [(lo, hi) for lo, hi, _, _ in got] == SH.bh_ranges(14, 4)
    assert all(js == 14 and sd == 3 for _, _, js, sd in got)
    # one GPU: both modes are the whole workload
    assert bench.rank_slices("weak", 16, 1, 0, 5) == bench.rank_slices("strong", 16, 1, 0, 5) == (0, 16, 16, 5)
