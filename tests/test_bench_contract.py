"""The JSON line bench.py prints: the keys and types the benchmark contract
fixes, for the reference arm (the CPU oracle: runs without a GPU) and for
this library's arm (GPU)."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

BASE_KEYS = {"metric": str, "value": float, "unit": str, "n_gpus": int, "steps": int, "warmup": int,
             "ms_per_step": float, "higher_is_better": bool, "scaling": str, "dtype": str, "data": str,
             "config": dict}


def run_bench(*args, timeout=600):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], cwd=ROOT,
                       capture_output=True, text=True, timeout=timeout)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [x for x in r.stdout.splitlines() if x.startswith("{")]
    assert len(lines) == 1, r.stdout[-2000:]
    return json.loads(lines[0])


def check_base(line):
    for k, t in BASE_KEYS.items():
        assert k in line, k
        assert isinstance(line[k], (int, float) if t is float else t), (k, line[k])
    assert line["higher_is_better"] is True and line["scaling"] == "weak"
    assert "vs_baseline" in line and line["vs_baseline"] is None
    assert isinstance(line["config"].get("workload"), str)
    assert line["value"] > 0 and line["ms_per_step"] > 0


def test_reference_arm_line():
    line = run_bench("--impl", "reference", "--steps", "1", "--warmup", "3")
    check_base(line)
    assert line["impl"] == "reference"
    cpu = line["cpu_baseline"]
    assert cpu["kind"] == "oracle" and cpu["cores"] >= 1 and cpu["value"] == line["value"]
    assert isinstance(cpu["sample"], str) and cpu["sample"]
    e2e = line["e2e"]
    assert e2e["value"] == line["value"] and e2e["unit"] == line["unit"]
    assert e2e["h2d_bytes_per_step"] == 0 and e2e["d2h_bytes_per_step"] == 0
    # the configuration is the workload's alone: the library arm prints the same dict
    sys.path.insert(0, ROOT)
    import bench
    from paper_2609_35352_gb300 import workloads as W
    assert line["config"] == bench.workload_config(W.make_workload(bench.DEFAULT_WORKLOAD),
                                                   bench.DEFAULT_WORKLOAD)
    assert line["config"]["bytes_min_per_step"] > 0 and "l2" in line["config"]


@pytest.mark.gpu
def test_library_arm_line():
    line = run_bench("--steps", "3", "--warmup", "3", "--no-cpu")
    check_base(line)
    assert line["n_gpus"] == 1 and line["gpu_launches"] == line["steps"]
    roof = line["roofline"]
    assert roof["bound"] == "hbm" and roof["unit"] == "GB/s"
    assert abs(roof["frac"] - roof["achieved"] / roof["peak"]) < 1e-9
    assert 0.3 < roof["frac"] < 1.3  # the default layer runs near the copy peak
    alu = line["alu"]
    assert alu["bound"] == "alu" and alu["peak"] > alu["achieved"] > 0
    e2e = line["e2e"]
    assert e2e["unit"] == line["unit"] and e2e["value"] > 0
    assert e2e["h2d_bytes_per_step"] > 0 and e2e["d2h_bytes_per_step"] > 0
    clk = line["clocks"]
    for k in ("sm_mhz", "sm_max_mhz", "reasons"):
        assert k in clk
    assert clk["samples"] >= 2 and clk["sm_mhz"] > 0  # taken inside the timed region
    assert roof["peak_nominal"] > roof["peak"] * 0.9 and 0 < roof["frac_nominal"] < roof["frac"] * 1.2
    ref = run_bench("--impl", "reference", "--steps", "1", "--warmup", "3")
    assert ref["config"] == line["config"]
