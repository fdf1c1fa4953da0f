"""bench.py's native arm as the multi-GPU launch runs it: two ranks under
torch.distributed.run, each stepping its own d-slice of one longer model
vector through the library (relay_set_coord_offset), a barrier and the max
over ranks around the timed region, one JSON line from rank 0.

One GPU is visible here, so the two ranks share it: bench.py then places
them round robin and runs the host collectives over gloo (NCCL refuses two
ranks on one device).  The ranks' kernels never wait on one another; only
the host barrier and the max-reduction cross ranks.  That the slices
reproduce the columns of one unsharded run is checked by
test_coordinate_offset_slice_equals_full_run."""
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


@pytest.mark.gpu
def test_native_arm_two_ranks_on_one_gpu():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py", "--gpus", "2",
           "--workload", "chain16_d9231114_dirichlet", "--steps", "3", "--warmup", "3",
           "--no-cpu-baseline", "--e2e-steps", "0", "--fused-steps", "0", "--no-per-workload"]
    env = dict(os.environ, CUDA_VISIBLE_DEVICES=os.environ.get("CUDA_VISIBLE_DEVICES", "0").split(",")[0],
               OMP_NUM_THREADS="1")
    out = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=900, env=env)
    assert out.returncode == 0, out.stderr[-3000:]
    lines = [json.loads(s) for s in out.stdout.splitlines() if s.startswith("{")]
    assert len(lines) == 1, out.stdout[-2000:]
    line = lines[0]
    assert line["n_gpus"] == 2 and line["steps"] == 3 and line["warmup"] == 3
    assert line["scaling"] == "weak" and line["unit"] == "steps/s" and line["value"] > 0
    assert line["gpu_launches"] == 2 * 2 * 3  # both ranks, counter + step kernel per step
    assert "share 1 GPU" in line["config"]["parallelism"]
    # the job's time is the slower rank's: value = 2 ranks x 3 steps over it
    assert abs(line["value"] - 2 * 3 / (line["ms_per_step"] * 3 / 1e3)) <= 1e-3 * line["value"]
    r = line["roofline"]
    assert r["bound"] == "hbm" and r["achieved"] > 0 and r["kernel"] == "relay_models_kernel"
    # the metrics of both ranks' slices, combined by the one all-reduce
    m = line["metrics"]
    assert m["coordinates"] == 2 * 9_231_114 and m["after_steps"] == 3 + 3
    assert 0 < m["consensus_distance"] < 10 and 0 < m["distance_to_optimum"] < 10


@pytest.mark.gpu
def test_native_arm_two_ranks_with_every_leg():
    """The legs the default command adds to the headline -- the per-workload
    lines, the several-steps-per-call rate and the host-state e2e step --
    run at two ranks too, with the same collectives on every rank, and rank 0
    prints one line that carries them all."""
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py", "--gpus", "2",
           "--workload", "chain16_d9231114_dirichlet", "--steps", "2", "--warmup", "3",
           "--no-cpu-baseline", "--e2e-steps", "1", "--fused-steps", "8"]
    env = dict(os.environ, CUDA_VISIBLE_DEVICES=os.environ.get("CUDA_VISIBLE_DEVICES", "0").split(",")[0],
               OMP_NUM_THREADS="1")
    out = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=1500, env=env)
    assert out.returncode == 0, out.stderr[-3000:]
    lines = [json.loads(s) for s in out.stdout.splitlines() if s.startswith("{")]
    assert len(lines) == 1, out.stdout[-2000:]
    line = lines[0]
    assert line["n_gpus"] == 2 and line["value"] > 0
    names = [p["workload"] for p in line["per_workload"]]
    assert "chain16_d9231114_dirichlet" not in names and len(names) >= 5, names
    for p in line["per_workload"]:
        assert p["value"] > 0 and p["roofline"]["frac"] > 0 and p["gpu_launches"] > 0, p
    f = line["fused_steps"]
    assert f["value"] > 0 and f["steps_per_call"] == 8
    e = line["e2e"]
    assert (e.get("value") or 0) > 0 or "skipped" in e, e
