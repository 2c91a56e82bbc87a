"""The benchmark harness on the host: the reference arm's JSON line (the
oracle on a small sample, no GPU), the clock-record summary and the DRAM
traffic lookup that fill the GPU arm's JSON line."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_reference_arm_prints_one_contract_line():
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                          "--warmup", "0", "--ref-sample-tokens", "512"], capture_output=True, text=True,
                         timeout=600, cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference"
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
              "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["value"] > 0 and d["unit"] == "tokens/s" and d["higher_is_better"] is True
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] == 1
    assert d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    assert "workload" in d["config"]


def test_clock_summary():
    rows = ["0, 2070, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active\n",
            "0, 2070, 2070, 1100.0, 0x4, Not Active, Not Active, Not Active, Active\n",
            "0, 1980, 2070, 1300.0, 0x0, Not Active, Not Active, Not Active, Not Active\n",
            "garbage\n"]
    c = bench.summarize_clock_lines(rows)
    assert c == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 3}
    hot = bench.summarize_clock_lines(["0, 1500, 2070, 1400, 0x8, Active, Not Active, Active, Not Active\n"])
    assert hot["reasons"] == ["hw_slowdown", "sw_thermal_slowdown"]
    assert bench.summarize_clock_lines([]) is None


def test_dram_traffic_lookup(tmp_path):
    p = tmp_path / "t.txt"
    p.write_text("# comment\nroute_topk 2097152 256 123\nmargin_hist_lei_pass2 2097152 256 456  # note\n")
    assert bench.dram_traffic(str(p), "margin_hist_lei_pass2", 2097152, 256) == 456
    assert bench.dram_traffic(str(p), "route_topk", 2097152, 128) is None
    assert bench.dram_traffic(str(tmp_path / "missing.txt"), "route_topk", 1, 1) is None


@pytest.mark.parametrize("kernel,T,E", [("margin_hist_lei_pass1", 2097152, 256),
                                        ("margin_hist_lei_pass2", 2097152, 256),
                                        ("router_route", 1048576, 128)])
def test_committed_traffic_covers_the_dominant_kernels(kernel, T, E):
    """The default and router workloads' dominant kernels have a recorded
    DRAM traffic figure, close to their algorithmic bytes."""
    path = os.path.join(ROOT, "profiles", "dram_traffic_per_launch.txt")
    v = bench.dram_traffic(path, kernel, T, E)
    assert v is not None
    alg = {"margin_hist_lei_pass1": 2 * T * E + 4 * T + 8 * (T // 2) * E,
           "margin_hist_lei_pass2": 2 * T * E + 4 * T + 8 * (T - T // 2) * E,
           "router_route": 2 * T * 4096 + 2 * E * 4096 + 2 * T * E + 4 * T * 8 + 4 * T}[kernel]
    assert 0.9 * alg <= v <= 1.05 * alg
