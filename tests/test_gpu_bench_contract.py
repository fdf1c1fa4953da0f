"""bench.py's native arm on one GPU: exactly one JSON line carrying every key
of the launch contract (throughput, roofline of the step kernel, the CPU
oracle baseline, the end-to-end rate through the host-state step, clocks,
kernel launches, metrics), on the 16-worker VGG-11-sized chain with a short
run."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.gpu
def test_native_line_carries_the_contract_keys():
    cmd = [sys.executable, "bench.py", "--workload", "chain16_d9231114_dirichlet", "--steps", "4",
           "--warmup", "3", "--e2e-steps", "2", "--fused-steps", "2", "--no-per-workload"]
    out = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=900)
    assert out.returncode == 0, out.stderr[-3000:]
    lines = [json.loads(s) for s in out.stdout.splitlines() if s.startswith("{")]
    assert len(lines) == 1, out.stdout[-2000:]
    j = lines[0]
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
              "scaling", "vs_baseline", "dtype", "data", "config", "roofline", "cpu_baseline", "e2e",
              "gpu_launches", "clocks", "metrics"):
        assert k in j, k
    assert j["n_gpus"] == 1 and j["steps"] == 4 and j["warmup"] == 3 and j["unit"] == "steps/s"
    assert j["higher_is_better"] is True and j["scaling"] == "weak" and j["dtype"] == "f32"
    assert j["vs_baseline"] is None and j["data"] == "synthetic"
    assert j["config"]["workload"] == "chain16_d9231114_dirichlet" and "l2" in j["config"]
    assert abs(j["value"] - 4 / (j["ms_per_step"] * 4 / 1e3)) <= 1e-3 * j["value"]
    r = j["roofline"]
    assert r["bound"] == "hbm" and r["unit"] == "GB/s" and r["peak"] > 0
    assert abs(r["frac"] - r["achieved"] / r["peak"]) < 1e-3
    assert r["algorithmic_bytes_per_launch"] == 4 * 9_231_114 * (2 * 16 + 2 * 30)
    assert r["traffic"] is None or r["traffic"] > r["algorithmic_bytes_per_launch"]
    assert r["launch_ms_mean"] <= j["ms_per_step"] * 1.001
    c = j["cpu_baseline"]
    assert c["kind"] == "oracle" and c["cores"] >= 1 and c["value"] > 0 and c["unit"] == "steps/s"
    assert "sample" in c
    e = j["e2e"]
    assert e["value"] > 0 and e["unit"] == "steps/s"
    assert e["h2d_bytes_per_step"] > 0 and e["d2h_bytes_per_step"] > 0
    # the state crosses the link every step: x, the message rows read, the counters in; x, every row out
    assert e["d2h_bytes_per_step"] == 4 * 9_231_116 * (16 + 30) + 4 * 30
    assert j["gpu_launches"] == 2 * 4
    clk = j["clocks"]
    assert clk is None or ("sm_mhz" in clk and "sm_max_mhz" in clk and "reasons" in clk)
    m = j["metrics"]
    assert m["after_steps"] == 3 + 4 and m["coordinates"] == 9_231_114
    assert 0 < m["consensus_distance"] and 0 < m["distance_to_optimum"]
    assert j["fused_steps"]["steps_per_call"] == 2 and j["fused_steps"]["value"] > 0
