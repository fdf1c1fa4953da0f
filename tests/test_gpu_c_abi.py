"""The C ABI driven from a C program (tests/c_abi_run.c: create, objective,
init, steps, allocation-free metrics, destroy), compiled against the
library, must give the same models bit for bit as the Python binding's run of
the same configuration, and the same metrics -- with the C program stepping
through relay_step calls, through one relay_steps call, or through
relay_step_host calls on a state in page-locked host memory."""
import os
import subprocess

import numpy as np
import pytest
import torch

import paper_2110_04175_gb300 as rs
from paper_2110_04175_gb300 import build as rs_build
from paper_2110_04175_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)


@pytest.fixture(scope="module")
def c_program(tmp_path_factory):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    lib = rs_build.build()
    exe = str(tmp_path_factory.mktemp("cabi") / "c_abi_run")
    subprocess.run(["nvcc", os.path.join(HERE, "c_abi_run.c"), "-I", os.path.join(ROOT, "include"),
                    "-L", os.path.dirname(lib), "-lrelaysum", "-o", exe], check=True)
    return exe, os.path.dirname(lib)


@pytest.mark.parametrize("path", ["step", "fused", "host"])
@pytest.mark.parametrize("tree,n,d,steps,mode", [("chain", 8, 4096, 100, 1), ("binary", 16, 70001, 30, 0)])
def test_c_program_equals_python_binding(c_program, tmp_path, tree, n, d, steps, mode, path):
    exe, libdir = c_program
    out = tmp_path / "out.bin"
    env = dict(os.environ, LD_LIBRARY_PATH=libdir + os.pathsep + os.environ.get("LD_LIBRARY_PATH", ""))
    r = subprocess.run([exe, tree, str(n), str(d), str(steps), str(mode), str(out)] + ([] if path == "step" else [path]),
                       env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr
    raw = out.read_bytes()
    x_c = np.frombuffer(raw[:4 * n * d], dtype=np.float32).reshape(n, d)
    m_c = np.frombuffer(raw[4 * n * d:], dtype=np.float64)

    edges = wl.chain(n) if tree == "chain" else wl.binary_tree(n)
    run = rs.RelayRun(n, d, edges, device="cuda:0", mode=mode)
    run.init(0.0, 0, wl.identity_mix(n), 2.0, 0, 0.1)
    for _ in range(steps):
        run.step(0.1, 0)
    m_py = run.metrics()[0].cpu().numpy()
    torch.cuda.synchronize()
    assert np.array_equal(x_c, run.x[:, :d].cpu().numpy())
    assert np.allclose(m_c, m_py, rtol=1e-12, atol=0)
