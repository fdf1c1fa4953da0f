"""The allocation-free metrics entry point (relay_metrics_static).

Some callers cannot allocate device memory -- code running while a CUDA
graph is captured in global mode, where cudaMalloc is refused, or a plug-in
whose host keeps all device memory in its own pool.  relay_metrics_static
serves them: it keeps its partial sums in scratch built into the library
instead of a caller workspace.  This test calls it through the C ABI twice in
a row, on models that change between the calls, and checks each result
against relay_metrics with an ordinary workspace: both run the same two
kernels with the same block count and the same fixed-order reduction, so
the results must be equal bit for bit.  It lives in a file that
pytest collects last, and it passes both alone and after the other tests.
"""
import numpy as np
import pytest
import torch

import paper_2110_04175_gb300 as rs
from paper_2110_04175_gb300 import build as rs_build
from paper_2110_04175_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    rs_build.build()


def test_static_scratch_metrics_equal_workspace_metrics_twice():
    n, d = 24, 1_000_003
    run = rs.RelayRun(n, d, wl.random_tree(n, 5), device="cuda:0")
    run.init(0.2, 1, wl.identity_mix(n), 1.5, 2, 0.1)
    h = run.h
    for call in range(2):
        for _ in range(3):
            run.step(0.1, 1)
        ws = torch.empty(rs.relay_metrics_workspace(h), dtype=torch.float64, device="cuda:0")
        want = torch.zeros(2, dtype=torch.float64, device="cuda:0")
        rs.relay_metrics(h, run.x, ws, want)
        got = torch.full((2,), float("nan"), dtype=torch.float64, device="cuda:0")
        rs.relay_metrics_static(h, run.x, got)
        torch.cuda.synchronize()
        g, w = got.cpu().numpy(), want.cpu().numpy()
        assert np.all(np.isfinite(g)) and np.all(w > 0), (call, g, w)
        assert torch.equal(got, want), (call, g, w)
