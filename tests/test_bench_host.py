"""Host-side logic of bench.py, on the CPU: the algorithmic byte counts that
the roofline fractions divide, the clock-record parsing that decides whether
a measurement stands, and the keying of the committed ncu traffic to the
kernel source it was taken on."""

import json
import os
import shutil

import numpy as np
import pytest

import bench


def test_algorithmic_bytes_hand_example():
    # B = 4, one mask word (N <= 63). Request 0: 10 tokens, 2 full blocks, reach 2
    # (probes both); request 1: 3 tokens, no block; request 2: 16 tokens, 4
    # blocks, reach 2 (probes blocks 0, 1 and the first miss, 2).
    lens = np.array([10, 3, 16], np.int64)
    local = np.array([4, 0, 8], np.int32)
    glob = np.array([4, 0, 0], np.int32)
    b = bench.algorithmic_bytes(lens, local, glob, 4, 1)
    assert b["k_digest"] == 4 * 4 * 6  # every token of the 6 full blocks
    assert b["k_probe"] == 5 * 16  # 2 + 0 + 3 probes, 16-byte entries
    assert b["k_chain"] == 16 * 6 + 24 * 3
    assert b["k_walk"] == 8 * 5 + 28 * 3
    assert b["k_prep"] == 16 * 3
    # 4 B per prompt token, an entry per probe, n + 1 offsets, 20 B of outputs per request
    assert b["path"] == 4 * 29 + 5 * 16 + 8 * 4 + 20 * 3


def test_algorithmic_bytes_probe_stops_after_the_first_miss():
    B, W = 32, 4
    lens = np.array([32 * 100 + 7] * 3, np.int64)
    local = np.array([0, 32 * 40, 32 * 100], np.int32)
    glob = np.array([0, 32 * 10, 0], np.int32)
    b = bench.algorithmic_bytes(lens, local, glob, B, W)
    assert b["k_probe"] == (1 + 51 + 100) * (8 + 8 * W)  # reach + 1, capped at n_r


def _sampler_with(rows):
    s = bench.ClockSampler("0")
    s.f.write("".join(r + "\n" for r in rows))
    return s.stop()  # never started: parses what the file holds


def test_clock_sampler_median_max_and_reasons():
    rows = [
        "0, 2070, 2070, 900.1, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
        "0, 1980, 2070, 1390.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
        "0, 2040, 2070, 1200.0, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
        "garbage line",
        "0, [N/A], 2070, 10.0, 0x0, Not Active, Not Active, Not Active, Not Active",
    ]
    c = _sampler_with(rows)
    assert c["sm_mhz"] == 2040 and c["sm_max_mhz"] == 2070
    assert c["reasons"] == ["sw_power_cap"] and c["samples"] == 3


def test_clock_sampler_reports_thermal_and_hw_slowdown():
    rows = ["0, 1500, 2070, 1000, 0x48, Active, Not Active, Active, Not Active"]
    c = _sampler_with(rows)
    assert c["reasons"] == ["hw_slowdown", "sw_thermal_slowdown"]


def test_clock_sampler_without_samples():
    c = _sampler_with([])
    assert c["sm_mhz"] is None and c["sm_max_mhz"] is None and c["samples"] == 0


@pytest.fixture()
def tree(tmp_path, monkeypatch):
    """A copy of the kernel sources and the traffic record that the test may edit."""
    csrc = tmp_path / "paper_2607_08565_gb300" / "csrc"
    csrc.mkdir(parents=True)
    for f in ("route.cu", "smetric_impl.cuh"):
        shutil.copy(os.path.join(bench.ROOT, "paper_2607_08565_gb300", "csrc", f), csrc / f)
    (tmp_path / "profiles").mkdir()
    shutil.copy(os.path.join(bench.ROOT, "profiles", "traffic.json"), tmp_path / "profiles" / "traffic.json")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    return tmp_path


def _section_bounds(text, section):
    banner = "// " + "-" * 75 + "\n"
    head = text.index("// " + section + "\n" + banner)
    start = head + len("// " + section + "\n" + banner)
    return start, text.index(banner, start)


def test_traffic_record_follows_the_digest_source(tree):
    rec = json.loads((tree / "profiles" / "traffic.json").read_text())["k_digest"]
    route = tree / "paper_2607_08565_gb300" / "csrc" / "route.cu"
    text = route.read_text()
    sha = bench.section_sha("digest")
    assert sha and len(sha) == 16
    assert bench.ncu_traffic("k_digest") == (rec["bytes_per_launch"] if sha == rec["source_sha"] else None)

    start, _ = _section_bounds(text, "digest")
    # comments and blank lines leave the kernel, and so its hash, unchanged
    route.write_text(text[:start] + "\n// a note about the digest\n\n" + text[start:])
    assert bench.section_sha("digest") == sha
    # a code change in the section gives another hash, and the record no longer applies
    route.write_text(text[:start] + "static const int kUnusedProbe = 1;\n" + text[start:])
    assert bench.section_sha("digest") != sha
    assert bench.ncu_traffic("k_digest") is None
    # as does a change to the shared device header
    route.write_text(text)
    hdr = tree / "paper_2607_08565_gb300" / "csrc" / "smetric_impl.cuh"
    hdr.write_text(hdr.read_text() + "\nstatic const int kUnusedHeader = 2;\n")
    assert bench.section_sha("digest") != sha
    assert bench.ncu_traffic("k_digest") is None


def test_traffic_record_missing_or_unknown(tree):
    assert bench.ncu_traffic("k_no_such_kernel") is None
    assert bench.section_sha("no such section") == ""
    os.unlink(tree / "profiles" / "traffic.json")
    assert bench.ncu_traffic("k_digest") is None


def test_peak_falls_back_only_without_a_measurement(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.peak_hbm() == (6800.0, "fallback")
    (tmp_path / "MEASURED_PEAKS.json").write_text(json.dumps({"hbm_gbs": 6798.6}))
    assert bench.peak_hbm() == (6798.6, "measured")
