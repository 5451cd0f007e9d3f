"""bench.py's host logic without a GPU: the clock summary of nvidia-smi samples, the L2
flush rule, the ncu-traffic lookup tied to the kernel sources, the measured peak, and
the bounded CPU-baseline sample of the oracle."""

import os
import shutil

import pytest

import bench
from synth import get_workload

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_clock_summary_median_and_reasons():
    lines = [
        "2070, 2070, 255.1, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
        "2055, 2070, 260.4, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
        "2070, 2070, 258.0, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
        "garbage line",
        "[N/A], 2070, 1.0, 0x0, Active, Not Active, Not Active, Not Active",
    ]
    c = bench.ClockSampler.summarise(lines)
    assert c["sm_mhz"] == 2070 and c["sm_max_mhz"] == 2070
    assert c["samples"] == 3 and c["power_w_max"] == 260.4
    assert c["reasons"] == ["hw_slowdown", "sw_power_cap"]   # a throttle seen with an unreadable clock counts
    hot = bench.ClockSampler.summarise(["1500, 2070, 900, 0x8, Not Active, Active, Not Active, Not Active"])
    assert hot["reasons"] == ["hw_thermal_slowdown"] and hot["sm_mhz"] == 1500
    assert bench.ClockSampler.summarise([])["reasons"] == ["no samples"]


def test_l2_flush_rule():
    small = get_workload("gpt2-small")
    assert bench.needs_l2_flush(small.weight_bytes() + 4 * small.layers * small.n_q * small.d)
    for name in ("gpt2-xl", "llama2-7b-planted", "llama2-70b-gqa"):
        wl = get_workload(name)
        assert not bench.needs_l2_flush(wl.weight_bytes() + 4 * wl.layers * wl.n_q * wl.d), name
    # the 4-layer profiling slice of the 70B shape is still larger than twice the L2
    assert not bench.needs_l2_flush(get_workload("llama2-70b-gqa").scaled(layers=4).weight_bytes())


def test_profiled_traffic_follows_the_kernel_source(tmp_path, monkeypatch):
    """bench.py reports the stored ncu traffic only while every listed source still has the
    hash the counters were taken on (checked on a copy of the tree)."""
    import hashlib
    import json
    csrc = tmp_path / "paper_2602_18851_gb300" / "csrc"
    csrc.mkdir(parents=True)
    for f in ("gas_gram.cu", "gas_device.cuh"):
        shutil.copy(os.path.join(ROOT, "paper_2602_18851_gb300", "csrc", f), csrc / f)
    sha = {f: hashlib.sha1((csrc / f).read_bytes()).hexdigest() for f in ("gas_gram.cu", "gas_device.cuh")}
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(
        {"gram_fused": {"unit": "layer", "bytes_per_unit": 1000, "sources": sha}}))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.profiled_traffic("gram_fused", 80) == 80000
    assert bench.profiled_traffic("gram_fused", 4) == 4000
    assert bench.profiled_traffic("writeback", 80) is None        # no figure kept
    with open(csrc / "gas_gram.cu", "a") as f:
        f.write("\n// edited\n")
    assert bench.profiled_traffic("gram_fused", 80) is None
    # the committed file parses, and every entry names its sources
    with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
        committed = json.load(f)
    for name, rec in committed.items():
        if not name.startswith("_"):
            assert rec["bytes_per_unit"] > 0 and rec["sources"], name


def test_measured_peak_is_read_from_the_driver_file():
    peak, kind = bench.measured_peaks()
    if os.path.exists(os.path.join(ROOT, "MEASURED_PEAKS.json")):
        assert kind == "measured" and 5000 < peak < 9000
    else:
        assert (peak, kind) == (6800.0, "fallback")


def test_cpu_baseline_sample_is_bounded_and_labelled():
    wl = get_workload("tiny-gqa128")
    c = bench.oracle_sample_ms(wl, wl.iters, budget_s=0.0)
    assert c["kind"] == "oracle" and c["unit"] == "ms" and c["cores"] >= 1 and c["value"] > 0
    assert "1 whole layers" in c["sample"] and wl.name in c["sample"]


def test_cpu_baseline_reports_all_cores_one_core_and_explicit():
    wl = get_workload("tiny-gqa128")
    c = bench.cpu_baseline(wl, wl.iters, budget_s=0.0)
    assert c["kind"] == "oracle" and c["value"] > 0 and c["cores"] >= 1
    assert c["single_thread"]["cores"] == 1 and c["single_thread"]["value"] > 0
    assert "1 thread" in c["single_thread"]["sample"]
    assert c["explicit"]["value"] > 0 and "explicitly formed" in c["explicit"]["sample"]
    # the one-thread run leaves the all-core figures alone: the explicit sample uses every core
    import oracle
    assert c["explicit"]["cores"] == c["cores"] == oracle.max_threads()
