"""Host-side logic of bench.py, on the CPU: the algorithmic byte counts that
the roofline fractions divide, the clock-record parsing that decides whether
a measurement stands, the keying of the committed ncu traffic to the
kernel source it was taken on, and the routed batches' hit and imbalance
statistics."""

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
    assert b["k_chain_probe"] == 16 * 6 + 24 * 3 + 5 * 16
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


def test_route_stats_hand_example():
    lens = [np.array([100, 50, 30, 20], np.int64), np.array([10, 10], np.int64)]
    outs = [dict(instance=np.array([0, 1, 0, 2], np.int32), local_hit=np.array([64, 0, 16, 0], np.int32),
                 global_hit=np.array([32, 48, 0, 0], np.int32)),
            dict(instance=np.array([1, 1], np.int32), local_hit=np.array([0, 0], np.int32),
                 global_hit=np.array([0, 0], np.int32))]
    s = bench.route_stats(lens, outs, 3)
    assert s["local_hit_ratio"] == 80 / 220 and s["global_hit_ratio"] == 80 / 220
    # batch 0: instance 0 gets 130 of 200 tokens; batch 1: one instance gets all 20
    assert s["routed_token_imbalance"] == pytest.approx((3 * 130 / 200 + 3.0) / 2)
    assert s["batches"] == 2
    empty = bench.route_stats([np.zeros(0, np.int64)], [dict(instance=np.zeros(0, np.int32),
                                                          local_hit=np.zeros(0, np.int32),
                                                          global_hit=np.zeros(0, np.int32))], 4)
    assert empty["local_hit_ratio"] == 0.0 and empty["routed_token_imbalance"] is None


def test_route_stats_on_oracle_routed_burst_batches():
    """The statistics of routed config-4-shaped batches (the oracle routes a
    reduced burst trace) lie in their ranges: hits within the prompts and an
    imbalance between 1 and N."""
    import oracle
    from synth import burst_trace
    oracle.build()
    tr = burst_trace(n_sessions=512, batch_size=64)
    p = tr.params
    host = [tr.batch(k) for k in range(2)]
    ox = bench.oracle_index_for(tr, host)
    outs = [ox.route_batch(p.block_size, p.session_blocks, p.hash_seed, b.tokens, b.offsets, b.load,
                           p.w_load, p.w_miss, p.w_glob) for b in host]
    ox.close()
    s = bench.route_stats([b.lengths() for b in host], outs, p.num_instances)
    assert 0.5 < s["local_hit_ratio"] + s["global_hit_ratio"] <= 1.0
    assert 1.0 <= s["routed_token_imbalance"] <= p.num_instances
    assert s["batches"] == 2


def test_cpu_baseline_reports_all_cores_and_one_thread():
    """The oracle timing the bench line carries: a bounded sample on the
    given cores and one on a single thread, each with its sample stated."""
    import oracle
    from synth import burst_trace
    oracle.build()
    tr = burst_trace(n_sessions=512, batch_size=64)
    bt = tr.batch(0)
    c = bench.cpu_baseline(tr, bt, 0, seconds=0.4, threads=2)
    assert c["kind"] == "oracle" and c["cores"] == 2 and c["unit"] == bench.UNIT
    assert c["value"] > 0 and c["tokens_per_s"] > 0 and "batch 0" in c["sample"]
    one = c["single_thread"]
    assert one["cores"] == 1 and one["value"] > 0 and "one thread" in one["sample"]
