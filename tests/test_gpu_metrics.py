"""Convergence metrics (relay_metrics): the consensus distance and the
distance of the average model to the optimum, as in the paper's analysis."""
import numpy as np
import pytest
import torch

import paper_2110_04175_gb300 as rs
from paper_2110_04175_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _reference(x, mu):
    x, mu = np.asarray(x, np.float64), np.asarray(mu, np.float64)
    xbar = x.mean(axis=0)
    return ((x - xbar) ** 2).sum(axis=0).mean() / x.shape[0], ((xbar - mu.mean(axis=0)) ** 2).mean()


@pytest.mark.parametrize("d", [1, 7, 1031, 300_001])
def test_metrics_match_float64_definition(d):
    n = 9
    run = rs.RelayRun(n, d, wl.random_tree(n, 1), device="cuda:0")
    run.init(0.3, 4, wl.identity_mix(n), 2.0, 5, 0.5)
    for _ in range(3):
        run.step(0.2, 4)
    m = run.metrics()[0].cpu().numpy()
    want = _reference(run.x[:, :d].cpu().numpy(), run.mu[:, :d].cpu().numpy())
    assert np.allclose(m, want, rtol=1e-9, atol=0)
    # deterministic: the same bits on every call
    assert np.array_equal(run.metrics()[0].cpu().numpy(), m)


def test_metrics_with_regenerated_centres_equal_stored():
    n, d = 16, 50_000
    mix = wl.dirichlet_mix(n, 10, 0.1, seed=1)
    out = []
    for objective in ("stored", "generated"):
        run = rs.RelayRun(n, d, wl.chain(n), device="cuda:0", objective=objective)
        run.init(0.1, 0, mix, 1.0, 2, 0.05)
        for _ in range(4):
            run.step(0.05, 0)
        out.append(run.metrics()[0].cpu().numpy())
    assert np.array_equal(out[0], out[1])


@pytest.mark.parametrize("scale", [1.0, 10.0])
@pytest.mark.parametrize("shape", ["chain", "star", "binary"])
def test_noise_free_runs_converge_linearly(shape, scale):
    """sigma = 0: both metrics fall geometrically to zero whatever the spread
    of the centres (appendix "Independence of heterogeneity")."""
    n, d = 16, 4096
    edges = {"chain": wl.chain(n), "star": wl.star(n), "binary": wl.binary_tree(n)}[shape]
    run = rs.RelayRun(n, d, edges, device="cuda:0")
    run.init(0.0, 0, wl.identity_mix(n), scale, 3, 0.0)
    run.step(0.3, 0)
    first = run.metrics()[0].cpu().numpy()
    for _ in range(400):
        run.step(0.3, 0)
    last = run.metrics()[0].cpu().numpy()
    assert last[0] < 1e-9 * first[0] and last[1] < 1e-9 * max(first[1], 1e-30) + 1e-20


@pytest.mark.parametrize("shape,n", [("chain", 16), ("binary", 16), ("star", 16), ("torus", 16)])
def test_lr_correction_matches_oracle(shape, n):
    from oracle import oracle
    edges = {"chain": wl.chain(n), "binary": wl.binary_tree(n), "star": wl.star(n),
             "torus": wl.torus_spanning_tree(4, 4, 0)}[shape]
    alpha, limits = rs.lr_correction(n, edges, mode=1, device="cuda:0")
    E = 2 * (n - 1)
    x, mu = np.zeros((n, 1)), np.ones((n, 1))
    msg, c = np.zeros((E, 1)), np.zeros(E, np.int32)
    oracle.run(n, edges, x, mu, msg, c, 1.0, 0.0, 0, 0, 1, 1)
    oracle.run(n, edges, x, mu, msg, c, 0.0, 0.0, 0, 1, 5000, 1)
    assert abs(alpha - x[:, 0].mean()) < 1e-5
    assert 0.0 < alpha < 1.0
