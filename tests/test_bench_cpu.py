"""Host-side pieces of bench.py, on CPU: the device-code hash that keys the
committed traffic capture (comment edits keep it, code edits void it), the
traffic lookup, the clock-log summary, the algorithmic byte count and the
workload overrides."""
import argparse
import json
import os
import shutil
import statistics
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2603_12707_gb300 import workloads as wl  # noqa: E402


def _copies(tmp_path):
    out = []
    for src in bench.KERNEL_SOURCES:
        dst = tmp_path / os.path.basename(src)
        shutil.copy(src, dst)
        out.append(str(dst))
    return out


def test_code_hash_ignores_comments_and_blank_lines(tmp_path):
    paths = _copies(tmp_path)
    h0 = bench.kernel_code_hash(paths)
    assert h0 == bench.kernel_code_hash(bench.KERNEL_SOURCES)
    with open(paths[0], "a") as f:
        f.write("\n\n// a new comment line\n   \n")
    s = open(paths[1]).read()
    open(paths[1], "w").write(s.replace("#pragma once", "#pragma once   // trailing comment", 1))
    assert bench.kernel_code_hash(paths) == h0


def test_code_hash_changes_with_code(tmp_path):
    paths = _copies(tmp_path)
    h0 = bench.kernel_code_hash(paths)
    s = open(paths[0]).read()
    assert "kWaitLimitNs = 1000000000ull" in s
    open(paths[0], "w").write(s.replace("kWaitLimitNs = 1000000000ull", "kWaitLimitNs = 1000000001ull", 1))
    assert bench.kernel_code_hash(paths) != h0


def test_traffic_lookup_needs_the_captured_code(tmp_path, monkeypatch):
    paths = _copies(tmp_path)
    prof = tmp_path / "profiles"
    prof.mkdir()
    rec = {"source_sha256_16": bench.kernel_code_hash(paths),
           "captures": {"qwen": {"traffic_over_algorithmic": 1.25}}}
    (prof / "decode_kernel_traffic.json").write_text(json.dumps(rec))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.committed_traffic(paths, "qwen", 1000) == 1250
    assert bench.committed_traffic(paths, "llava", 1000) is None      # no capture for it
    s = open(paths[0]).read()
    open(paths[0], "w").write(s.replace("kWaitLimitNs = 1000000000ull", "kWaitLimitNs = 2000000000ull", 1))
    assert bench.committed_traffic(paths, "qwen", 1000) is None       # code changed since


def test_clock_summary_reads_the_nvidia_smi_log(tmp_path):
    log = tmp_path / "clocks.csv"
    log.write_text(
        "0, 2070, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active\n"
        "0, 1980, 2070, 1350.0, 0x4, Not Active, Not Active, Not Active, Active\n"
        "0, 2070, 2070, 1390.2, 0x4, Not Active, Not Active, Not Active, Active\n"
        "garbage line\n")
    c = bench.ClockSampler(0)
    c.proc, c.path = object(), str(log)
    s = c.summary()
    assert s == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 3}
    assert not log.exists()


def test_layer_bytes_closed_form():
    cfg = wl.CONFIGS["qwen"]
    attended = [1, 17, 300]
    attn, app = bench.layer_bytes(cfg, attended)
    kv = sum(attended) * 2 * 4 * 128 * 2
    assert attn == kv + 3 * 28 * 128 * 2 * 2
    assert app == 3 * 2 * 4 * 128 * 2


def test_workload_overrides():
    a = argparse.Namespace(config="qwen", phys_layers=0, page_order=None)
    assert bench.workload_config(a) == wl.CONFIGS["qwen"]
    a = argparse.Namespace(config="qwen", phys_layers=4, page_order="shuffled")
    cfg = bench.workload_config(a)
    assert (cfg.phys_layers, cfg.page_order, cfg.num_layers) == (4, "shuffled", 28)
    assert bench.describe(cfg)["page_order"] == "shuffled"


def test_clock_records_the_timing_rules_reject():
    ok = {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": [], "samples": 5}
    cap = {"sm_mhz": 1800.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 5}
    assert not bench.clocks_slowed(ok)
    assert not bench.clocks_slowed(cap)              # the power cap is kept and noted
    for r in ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"):
        assert bench.clocks_slowed({**ok, "reasons": [r]})
    assert bench.clocks_slowed({**ok, "sm_mhz": 1200.0})   # far below max with no reason: a clock lock
    assert not bench.clocks_slowed({"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0})


def test_timed_blocks_cover_the_target_time_within_bounds():
    ns = argparse.Namespace(block_target_s=0.5, min_blocks=3, max_blocks=10)
    assert bench.block_count(94.0, ns) == 6         # 6 x 94 ms >= 0.5 s
    assert bench.block_count(11.0, ns) == 10        # capped
    assert bench.block_count(1080.0, ns) == 3       # at least 3
    assert bench.block_count(0.0, ns) == 10


def test_median_block_is_the_middle_of_the_sorted_times():
    assert bench.median_block([5.0, 1.0, 3.0]) == 2
    assert bench.median_block([4.0, 1.0, 3.0, 2.0]) == 3    # lower median: 2.0
    assert bench.median_block([7.0]) == 0


def _fake_run(cfg, block_ms, steps, L):
    """A run record as run_gpu returns it: blocks of `steps` steps whose
    attended lengths grow by one per step."""
    blocks = []
    lens = [100, 200]
    for ms in block_ms:
        step_bytes, attn_bytes = [], []
        for _ in range(steps):
            att = [n + 1 for n in lens]
            a, p = bench.layer_bytes(cfg, att)
            step_bytes.append(L * (a + p))
            attn_bytes.append(a + p)
            lens = [n + 1 for n in lens]
        blocks.append({"ms": ms, "step_ms": [ms / steps] * steps, "attn_ms": [0.9 * ms / steps / L] * steps,
                       "step_bytes": step_bytes, "attn_bytes": attn_bytes,
                       "attended": [150.5 + len(blocks) * steps + i for i in range(steps)],
                       "kv_bytes": [L * bench.kv_bytes(cfg, [101 + len(blocks) * steps + i, 201 + len(blocks) * steps + i])
                                    for i in range(steps)]})
    clocks = {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": [], "samples": 12, "retimed": False}
    e2e = {"ms": 1.1 * sum(block_ms) / len(block_ms), "wall_s": 0.1, "bytes": sum(blocks[0]["step_bytes"]),
           "h2d": 1000, "d2h": 500}
    return {"blocks": blocks, "launches": 3 * steps, "clocks": clocks, "e2e": e2e, "cfg": cfg, "L": L,
            "start_attended": 151.0}


def test_summary_reports_the_median_block_and_every_contract_key():
    import dataclasses
    cfg = dataclasses.replace(wl.custom("fake", 2, 8, 8, 64, 2, lens=[100, 200], seed=1), phys_layers=2)
    steps, L = 4, 2
    ns = argparse.Namespace(steps=steps, config="tiny", page_order=None, unfused=False, split_pages=0, graph=True)
    r = _fake_run(cfg, [3.0, 1.0, 2.0], steps, L)
    out = bench.summarize(ns, 1, r)
    mid = r["blocks"][2]                       # 2.0 ms is the median of 3.0, 1.0, 2.0
    assert out["ms_per_step"] == round(2.0 / steps, 4)
    assert out["value"] == round(sum(mid["step_bytes"]) / 2.0e-3 / 1e9, 2)
    assert out["steps_per_s"] == round(steps / 2.0e-3, 3)
    assert out["timed_blocks"] == 3 and out["block_ms"] == [3.0, 1.0, 2.0]
    all_gbs = sum(sum(b["step_bytes"]) for b in r["blocks"]) / 6.0e-3 / 1e9
    assert out["all_blocks_gbs"] == round(all_gbs, 2)
    ro = out["roofline"]
    assert set(ro) >= {"bound", "achieved", "peak", "unit", "frac", "traffic"}
    assert ro["bound"] == "hbm" and ro["unit"] == "GB/s"
    assert abs(ro["frac"] - ro["achieved"] / ro["peak"]) < 1e-3
    assert out["e2e"]["h2d_bytes_per_step"] == 1000 and out["e2e"]["d2h_bytes_per_step"] == 500
    assert out["e2e"]["unit"] == "GB/s" and out["e2e"]["value"] > 0
    assert out["clocks"]["samples"] == 12 and out["gpu_launches"] == 3 * steps
    assert out["config"]["workload"].startswith("fake") and "l2" in out["config"]
    # the median block (the third) attends 158.5 .. 161.5 tokens on average over its steps
    ctx = out["median_block_context"]
    assert ctx["mean_attended_tokens"] == 160.0
    assert ctx["tokens_appended_before_it"] == 9
    kv = statistics.mean(L * bench.kv_bytes(cfg, [109 + i, 209 + i]) for i in range(steps))
    assert ctx["kv_gb_per_step"] == round(kv / 1e9, 4)
