"""Host-side logic of bench.py that needs no GPU: the clock record taken from
nvidia-smi samples (fed fake CSV lines here), the DRAM-traffic figure read
from a committed ncu summary only while its source hash matches, and the
role names given to the forward's GEMM launch records."""
import hashlib
import os

import bench


def _row(clock, power, hw=False, thermal=False, sw_thermal=False, power_cap=False):
    flag = lambda on: "Active" if on else "Not Active"
    return (f"0, {clock}, 2070, {power}, 0x0, {flag(hw)}, {flag(thermal)}, {flag(sw_thermal)}, "
            f"{flag(power_cap)}")


def test_clock_summary_median_under_load_and_reasons():
    lines = [_row(1200, 90.0), _row(2070, 1100.0), _row(2040, 1250.0, power_cap=True), _row(2010, 1200.0),
             "garbage line", ""]
    rec = bench.summarize_clock_rows(lines)
    assert rec["samples"] == 4
    assert rec["sm_mhz"] == 2040.0  # median of the three samples above 300 W
    assert rec["sm_max_mhz"] == 2070.0
    assert rec["reasons"] == ["sw_power_cap"]
    assert rec["power_w_max"] == 1250.0


def test_clock_summary_reports_every_slowdown_seen():
    lines = [_row(1800, 900.0, hw=True), _row(1700, 950.0, thermal=True, sw_thermal=True)]
    assert bench.summarize_clock_rows(lines)["reasons"] == ["hw_slowdown", "hw_thermal_slowdown",
                                                            "sw_thermal_slowdown"]


def test_clock_summary_idle_or_unparsable_samples():
    # no sample above 300 W: the median is over all samples
    assert bench.summarize_clock_rows([_row(1000, 80.0), _row(1100, 90.0)])["sm_mhz"] == 1050.0
    # a sample whose clock field does not parse does not shift the others
    rec = bench.summarize_clock_rows([_row("[N/A]", 1000.0), _row(2000, 1000.0)])
    assert rec["sm_mhz"] == 2000.0
    assert bench.summarize_clock_rows([])["reasons"] == ["no samples"]


def test_committed_traffic_only_for_the_captured_source(tmp_path, monkeypatch):
    src = tmp_path / "kernel.cu"
    hdr = tmp_path / "kernel.cuh"
    src.write_bytes(b"__global__ void k() {}\n")
    hdr.write_bytes(b"#pragma once\n")
    sha = hashlib.sha256(src.read_bytes() + hdr.read_bytes()).hexdigest()
    assert bench.source_sha256([str(src), str(hdr)]) == sha
    prof = tmp_path / "profiles"
    prof.mkdir()
    (prof / "k.md").write_text("notes\n\ntraffic_kernel: k_kernel traffic_bytes_per_launch: 12.5e6 "
                               f"source_sha256: {sha}\n")
    (prof / "ignored.ncu-rep").write_text(f"traffic_kernel: k_kernel traffic_bytes_per_launch: 1 source_sha256: {sha}")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    files = [str(src), str(hdr)]
    assert bench.committed_traffic("k_kernel", files) == 12.5e6
    assert bench.committed_traffic("other_kernel", files) is None
    hdr.write_bytes(b"#pragma once  // changed\n")  # any of the kernel's sources changing voids the figure
    assert bench.committed_traffic("k_kernel", files) is None


def test_committed_traffic_without_profiles(tmp_path, monkeypatch):
    src = tmp_path / "kernel.cu"
    src.write_bytes(b"x")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.committed_traffic("k_kernel", [str(src)]) is None


def test_gemm_records_named_by_role():
    recs = [{"kind": "patchify", "layer": -1}, {"kind": "gemm", "layer": -1}]
    for layer in range(2):
        recs += [{"kind": "layernorm", "layer": layer}, {"kind": "gemm", "layer": layer},
                 {"kind": "attention", "layer": layer}, {"kind": "gemm", "layer": layer},
                 {"kind": "layernorm", "layer": layer}, {"kind": "gemm", "layer": layer},
                 {"kind": "gemm", "layer": layer}]
    recs.append({"kind": "head", "layer": -1})
    names = [n for n, _ in bench.label_records(recs)]
    assert names[:2] == ["patchify", "gemm.patch"]
    assert names[2:9] == ["layernorm", "gemm.qkv", "attention", "gemm.proj", "layernorm", "gemm.fc1", "gemm.fc2"]
    assert names[9:16] == names[2:9]
    assert names[-1] == "head"
    assert os.path.basename(bench.__file__) == "bench.py"
