"""bench.py's launch contract, exercised on CPU through its reference arm
(the CPU oracle): one process, and two ranks under torch.distributed.run as
the multi-GPU launch uses them.  Exactly one JSON line must come out (rank 0
only), carrying the keys the contract names."""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _json_lines(out: str):
    return [json.loads(line) for line in out.splitlines() if line.startswith("{")]


def _check_reference_line(line, gpus):
    assert line["impl"] == "reference"
    assert line["n_gpus"] == gpus and line["steps"] == 1 and line["warmup"] == 3
    assert line["value"] > 0 and line["unit"] == "steps/s" and line["higher_is_better"] is True
    assert line["config"]["workload"] == "chain8_d4096"
    cpu = line["cpu_baseline"]
    assert cpu["kind"] == "oracle" and cpu["cores"] >= 1 and cpu["value"] == line["value"]
    assert "sample" in cpu
    e2e = line["e2e"]
    assert e2e["value"] == line["value"] and e2e["h2d_bytes_per_step"] == 0
    assert e2e["d2h_bytes_per_step"] == 0


ARGS = ["--impl", "reference", "--steps", "1", "--warmup", "3", "--workload", "chain8_d4096"]


def test_reference_arm_one_process():
    out = subprocess.run([sys.executable, "bench.py", *ARGS], cwd=ROOT, capture_output=True, text=True,
                         timeout=600)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = _json_lines(out.stdout)
    assert len(lines) == 1
    _check_reference_line(lines[0], 1)


def test_reference_arm_two_ranks_under_torchrun():
    """As the driver launches N > 1: every rank exits 0, rank 0 alone prints."""
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py", "--gpus", "2", *ARGS]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    out = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=900, env=env)
    assert out.returncode == 0, out.stderr[-3000:]
    lines = _json_lines(out.stdout)
    assert len(lines) == 1
    _check_reference_line(lines[0], 2)


def test_warmup_below_three_is_refused():
    out = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--warmup", "2"], cwd=ROOT,
                         capture_output=True, text=True, timeout=300)
    assert out.returncode != 0 and "--warmup" in out.stderr


if __name__ == "__main__":
    sys.exit(pytest.main([__file__, "-q"]))


def test_traffic_entries_cover_the_default_line():
    """Every workload of the default bench line (the headline and its
    per-workload entries, all on the walk with stored centres) has a committed
    ncu DRAM-traffic figure, so the line's roofline.traffic is never null
    for a missing entry; the figures are of the order of the algorithmic bytes."""
    sys.path.insert(0, ROOT)
    import bench
    from paper_2110_04175_gb300 import workloads as wl
    for name in [bench.DEFAULT_WORKLOAD] + bench.PER_WORKLOAD:
        w = wl.by_name(name)
        t = bench.traffic_per_launch(w, "stored", "relay_models_kernel", "sgd")
        assert t is not None, name
        assert 0.8 < t / w.bytes_per_step() < 1.3, (name, t, w.bytes_per_step())
