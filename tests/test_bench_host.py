"""Host logic of bench.py, on the CPU: the clock record (parsed from canned
nvidia-smi lines in place of the tool), the source stamp that keeps the
stored DRAM-traffic figure tied to the kernel it was measured on, and the
peak used as the roofline denominator."""
import json
import os
import shutil
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2607_23089_gb300 import build as bld  # noqa: E402


def _sampler(lines):
    c = bench.ClockSampler(0)
    c.out = "\n".join(lines)
    return c


def test_clock_summary_median_max_and_reasons():
    lines = ["0, 2070, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active",
             "0, 1965, 2070, 1399.0, 0x4, Not Active, Not Active, Not Active, Active",
             "0, 2070, 2070, 1100.5, 0x0, Not Active, Not Active, Not Active, Not Active",
             "garbage line", "0, n/a, 2070, 0, 0, a, b, c, d"]
    s = _sampler(lines).summary()
    assert s["sm_mhz"] == 2070.0 and s["sm_max_mhz"] == 2070.0 and s["samples"] == 3
    assert s["reasons"] == ["sw_power_cap"]
    hot = _sampler(["0, 1500, 2070, 1400, 0x48, Active, Active, Not Active, Not Active"]).summary()
    assert hot["reasons"] == ["hw_slowdown", "hw_thermal_slowdown"]


def test_clock_summary_without_samples():
    s = _sampler([]).summary()
    assert s["samples"] == 0 and s["reasons"] == ["unavailable"] and s["sm_mhz"] is None


def _copy_tree(tmp_path, monkeypatch):
    """A copy of the kernel sources at another path, with the build module
    pointed at it as a checkout there would be."""
    root = tmp_path / "elsewhere"
    shutil.copytree(bld.CSRC, root / "paper_2607_23089_gb300" / "csrc")
    shutil.copytree(bld.INCLUDE, root / "include")
    csrc = str(root / "paper_2607_23089_gb300" / "csrc")
    inc = str(root / "include")
    flags = [csrc if f == bld.CSRC else inc if f == bld.INCLUDE else f for f in bld.NVCC_FLAGS]
    monkeypatch.setattr(bld, "ROOT", str(root))
    monkeypatch.setattr(bld, "CSRC", csrc)
    monkeypatch.setattr(bld, "INCLUDE", inc)
    monkeypatch.setattr(bld, "NVCC_FLAGS", flags)
    return csrc


def test_stamp_does_not_depend_on_the_checkout_path(tmp_path, monkeypatch):
    here = bench.headline_kernel_stamp()
    _copy_tree(tmp_path, monkeypatch)
    assert bench.headline_kernel_stamp() == here


def test_stamp_follows_the_headline_sources_only(tmp_path, monkeypatch):
    csrc = _copy_tree(tmp_path, monkeypatch)
    base = bench.headline_kernel_stamp()
    with open(os.path.join(csrc, "bwd_row.cuh"), "a") as f:  # not the headline kernel
        f.write("\n// edited\n")
    assert bench.headline_kernel_stamp() == base
    with open(os.path.join(csrc, "tile_row.cuh"), "a") as f:
        f.write("\n// edited\n")
    assert bench.headline_kernel_stamp() != base


def test_traffic_is_dropped_once_its_kernel_changes(tmp_path, monkeypatch):
    rec = os.path.join(ROOT, "profiles", "fused_ragged_layernorm_traffic.json")
    with open(rec) as f:
        stored = json.load(f)
    csrc = _copy_tree(tmp_path, monkeypatch)
    expect = stored["traffic_bytes_per_launch"]
    if stored["source_stamp"] != bench.headline_kernel_stamp():
        expect = None  # the record is of other sources: nothing is reported
    assert bench.profile_traffic() == expect
    with open(os.path.join(csrc, "small_row.cuh"), "a") as f:
        f.write("\n// edited\n")
    assert bench.profile_traffic() is None


def test_peak_is_measured_or_the_stated_fallback(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.peaks() == (bench.FALLBACK_HBM_GBS, "fallback")
    (tmp_path / "MEASURED_PEAKS.json").write_text(json.dumps({"hbm_gbs": 6698.5}))
    assert bench.peaks() == (6698.5, "measured")


if __name__ == "__main__":
    pytest.main([__file__, "-q"])
