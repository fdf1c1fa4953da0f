"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test would fail on a plausible mistake in the oracle: a wrong Philox
round, a swapped Box-Muller output, a counter that counts the receiver, a
message that includes the edge it is sent on, a rebuild that misses a term.
"""
import math
import os

import numpy as np
import pytest
from scipy import stats

from oracle import oracle
from paper_2110_04175_gb300 import workloads as wl
from tests import treeutil as tu

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ------------------------------------------------------------ random numbers

def test_philox_known_answers():
    """Philox4x32-10 reproduces the published known-answer vectors."""
    rows = []
    with open(os.path.join(GOLDEN, "philox4x32_10_kat.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                rows.append([int(v, 16) for v in line.split()])
    assert len(rows) == 3
    for r in rows:
        assert oracle.philox4x32_10(r[0:4], r[4:6]) == tuple(r[6:10])


def test_uniform_map_exact_range():
    """u = ((w >> 8) + 1) 2^-24: the 24 high bits, in (0, 1], never 0."""
    assert oracle.uniform(0) == 2.0 ** -24
    assert oracle.uniform(0xFF) == 2.0 ** -24
    assert oracle.uniform(0x100) == 2.0 * 2.0 ** -24
    assert oracle.uniform(0xFFFFFFFF) == 1.0
    assert oracle.uniform(0x80000000) == 0.5 + 2.0 ** -24


def test_box_muller_outputs_are_standard_normal():
    """Every one of the four outputs of a block is N(0, 1) (Kolmogorov-Smirnov),
    and the two outputs of one Box-Muller pair are uncorrelated."""
    nq = 12000
    z = oracle.normals(seed=12345, c0=0, length=4 * nq, row=3, step=7, stream=0).reshape(nq, 4)
    for r in range(4):
        col = z[:, r]
        assert abs(col.mean()) < 0.05
        assert abs(col.std() - 1.0) < 0.03
        assert stats.kstest(col, "norm").pvalue > 1e-3, r
    assert abs(np.corrcoef(z[:, 0], z[:, 1])[0, 1]) < 0.05
    assert abs(np.corrcoef(z[:, 2], z[:, 3])[0, 1]) < 0.05
    assert abs(np.corrcoef(z[:, 0], z[:, 2])[0, 1]) < 0.05


def test_vector_normals_equal_one_call_per_coordinate():
    """oracle.normals (one C loop) returns exactly oracle_normal per coordinate."""
    lib = oracle._load()
    for seed, c0, row, step, stream in ((0, 0, 0, 0, 0), (99, 37, 5, 3, 0), (2**40 + 7, 1001, 31, 49, 1)):
        got = oracle.normals(seed, c0, 67, row=row, step=step, stream=stream)
        want = np.array([lib.oracle_normal(seed, c0 + c, row, step, stream) for c in range(67)])
        assert np.array_equal(got, want)


def test_streams_rows_steps_differ():
    base = oracle.normals(7, 0, 64, row=0, step=0, stream=0)
    for kw in (dict(row=1, step=0, stream=0), dict(row=0, step=1, stream=0),
               dict(row=0, step=0, stream=1)):
        other = oracle.normals(7, 0, 64, **kw)
        assert abs(np.corrcoef(base, other)[0, 1]) < 0.5
        assert not np.allclose(base, other)


# ------------------------------------------------------------------- trees

@pytest.mark.parametrize("edges,n", [
    ([(0, 1), (1, 2), (2, 0)], 4),        # wrong edge count
    ([(0, 1), (1, 2), (0, 1)], 4),        # duplicate
    ([(0, 0), (1, 2), (2, 3)], 4),        # self loop
    ([(0, 1), (2, 3), (3, 2)], 4),        # disconnected / duplicate
    ([(0, 1), (1, 2), (2, 4)], 4),        # out of range
    ([(0, 1), (1, 2), (2, 0)], 3),        # cycle
])
def test_rejects_non_trees(edges, n):
    with pytest.raises(oracle.OracleError) as e:
        oracle.edges(n, edges)
    assert e.value.status == oracle.ORACLE_ENOTTREE


def test_directed_edge_numbering():
    edges = [(2, 0), (0, 1), (1, 3)]
    src, dst = oracle.edges(4, edges)
    assert list(zip(src, dst)) == tu.directed(edges)


# ---------------------------------------------------------------- counters

def _run_counts(n, edges, steps):
    """Counters after each step t = 0..steps-1, and nbar^{t+1}."""
    E = 2 * len(edges)
    counts = np.zeros(E, dtype=np.int32)
    empty = np.zeros((n, 0))
    out = []
    for t in range(steps):
        nbar = oracle.run(n, edges, empty, empty.copy(), np.zeros((E, 0)), counts, 0.0, 0.0, 0,
                          t, 1, 0)
        out.append((counts.copy(), nbar.copy()))
    return out


@pytest.mark.parametrize("n", [1, 2, 3, 4, 5, 6])
def test_counts_closed_form_every_tree(n):
    """c^t_{i->j} = |{l in T_{i\\j} : tau_il <= t}| and nbar^{t+1}_i = |{l : tau_il <= t+1}|
    at every step, for every labelled tree with n nodes.  Once t >= diam - 1 every
    counter is the size of the subtree behind its edge, and nbar = n once
    t + 1 >= ecc(i) (Alg. 1: nbar converges to the number of workers)."""
    for edges in tu.all_trees(n):
        tau = tu.distances(n, edges)
        diam = tu.diameter(n, edges)
        dedges = tu.directed(edges)
        sides = [tu.side(n, edges, i, j) for (i, j) in dedges]
        for t, (c, nbar) in enumerate(_run_counts(n, edges, diam + 2)):
            for e, (i, j) in enumerate(dedges):
                want = sum(1 for l in sides[e] if tau[i][l] <= t)
                assert c[e] == want, (edges, t, e)
                if t >= diam - 1:
                    assert c[e] == len(sides[e])
            for i in range(n):
                assert nbar[i] == sum(1 for l in range(n) if tau[i][l] <= t + 1)
                if t + 1 >= max(tau[i]):
                    assert nbar[i] == n


# ------------------------------------------------- messages with x held fixed

@pytest.mark.parametrize("n", [2, 3, 4, 5, 6])
def test_messages_sum_subtrees_with_fixed_models(n):
    """With gamma = sigma = 0 and the models reset to the same integer vector
    before every step, m^t_{i->j} is the exact sum of x over the nodes of
    T_{i\\j} within t hops of i; after diam - 1 steps, over the whole subtree."""
    rng = np.random.default_rng(n)
    trees = list(tu.all_trees(n))
    if len(trees) > 200:
        trees = [trees[k] for k in rng.choice(len(trees), 200, replace=False)]
    L = 3
    for edges in trees:
        E = 2 * len(edges)
        tau = tu.distances(n, edges)
        diam = tu.diameter(n, edges)
        dedges = tu.directed(edges)
        x_fixed = rng.integers(-50, 50, size=(n, L)).astype(np.float64)
        mu = np.zeros((n, L))
        msg = np.zeros((E, L))
        counts = np.zeros(E, dtype=np.int32)
        for t in range(diam + 1):
            x = x_fixed.copy()
            oracle.run(n, edges, x, mu, msg, counts, 0.0, 0.0, 0, t, 1, 0)
            for e, (i, j) in enumerate(dedges):
                members = [l for l in tu.side(n, edges, i, j) if tau[i][l] <= t]
                want = x_fixed[members].sum(axis=0)
                assert np.array_equal(msg[e], want), (edges, t, e)
        for e, (i, j) in enumerate(dedges):
            assert np.array_equal(msg[e], x_fixed[sorted(tu.side(n, edges, i, j))].sum(axis=0))


# --------------------------------------------------------- constant models

@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("shape", ["chain", "binary", "star", "random"])
def test_zero_gradient_keeps_models_constant(mode, shape):
    """Identical x^0 and zero gradients (gamma = 0, or mu_i = x^0 and sigma = 0):
    every model stays x^0.  Exact for dyadic x^0."""
    n = 9
    edges = {"chain": wl.chain(n), "binary": wl.binary_tree(n), "star": wl.star(n),
             "random": wl.random_tree(n, 3)}[shape]
    L = 16
    x0 = (np.arange(L) - 7.0) / 8.0
    for lr, mu in ((0.0, np.random.default_rng(0).normal(size=(n, L))), (0.3, np.tile(x0, (n, 1)))):
        x = np.tile(x0, (n, 1))
        msg = np.zeros((2 * (n - 1), L))
        counts = np.zeros(2 * (n - 1), dtype=np.int32)
        oracle.run(n, edges, x, mu, msg, counts, lr, 0.0, 0, 0, 25, mode)
        assert np.array_equal(x, np.tile(x0, (n, 1)))


def test_zero_gradient_random_x0_within_ulps():
    n = 7
    edges = wl.random_tree(n, 5)
    x0 = np.random.default_rng(1).normal(size=32)
    x = np.tile(x0, (n, 1))
    oracle.run(n, edges, x, np.zeros((n, 32)), np.zeros((12, 32)), np.zeros(12, dtype=np.int32),
               0.0, 0.0, 0, 0, 20, 0)
    assert np.max(np.abs(x - x0) / np.abs(x0)) < 8 * np.finfo(np.float64).eps


# ------------------------------------------------------------ special cases

def test_single_worker_is_plain_sgd():
    """n = 1: no edges, nbar = 1, so x^{t+1} = x^t - gamma((x^t - mu) + sigma xi^t);
    with sigma = 0, x^T = mu + (1 - gamma)^T (x^0 - mu)."""
    L = 8
    mu = np.linspace(-1, 1, L)[None, :]
    x = np.full((1, L), 3.0)
    lr = 0.25
    oracle.run(1, np.zeros((0, 2), np.int32), x, mu, np.zeros((0, L)), np.zeros(0, np.int32),
               lr, 0.0, 0, 0, 10, 0)
    want = mu + (1 - lr) ** 10 * (3.0 - mu)
    assert np.allclose(x, want, rtol=1e-14, atol=1e-14)


def test_noise_wiring_single_step():
    """With mu = x^0 = 0 and gamma = 1, one step gives x^1 = -sigma xi^0 with
    xi the stream-0 normal of row 0, step 0 (and of step t at step t)."""
    L = 12
    for t in (0, 5):
        x = np.zeros((1, L))
        oracle.run(1, np.zeros((0, 2), np.int32), x, np.zeros((1, L)), np.zeros((0, L)),
                   np.zeros(0, np.int32), 1.0, 0.5, 99, t, 1, 0, c0=40)
        want = -0.5 * oracle.normals(99, 40, L, row=0, step=t, stream=0)
        assert np.allclose(x[0], want, rtol=0, atol=1e-15)


@pytest.mark.parametrize("mode", [0, 1])
def test_two_workers_are_allreduce_sgd(mode):
    """n = 2: one edge, nbar = 2 from the first step, so both workers hold the
    all-reduce average (x_0^{t+1/2} + x_1^{t+1/2}) / 2 after every step."""
    L = 10
    rng = np.random.default_rng(2)
    mu = rng.normal(size=(2, L))
    x = np.tile(rng.normal(size=L), (2, 1))
    msg = np.zeros((2, L))
    counts = np.zeros(2, np.int32)
    lr, sigma, seed = 0.2, 0.3, 5
    for t in range(6):
        xh = np.empty_like(x)
        for i in range(2):
            xi = oracle.normals(seed, 0, L, row=i, step=t, stream=0)
            xh[i] = x[i] - lr * ((x[i] - mu[i]) + sigma * xi)
        oracle.run(2, [(0, 1)], x, mu, msg, counts, lr, sigma, seed, t, 1, mode)
        avg = (xh[0] + xh[1]) / 2
        assert np.allclose(x[0], avg, rtol=1e-13, atol=1e-13)
        assert np.allclose(x[1], avg, rtol=1e-13, atol=1e-13)


def test_star_hub_is_allreduce_every_step():
    """On a star the hub receives every leaf's x^{t+1/2} directly, so it holds
    the exact all-reduce average at every step."""
    n, L = 6, 8
    rng = np.random.default_rng(3)
    mu = rng.normal(size=(n, L))
    x = np.zeros((n, L))
    E = 2 * (n - 1)
    msg = np.zeros((E, L))
    counts = np.zeros(E, np.int32)
    lr, sigma, seed = 0.1, 0.2, 11
    for t in range(5):
        xh = np.array([x[i] - lr * ((x[i] - mu[i]) + sigma * oracle.normals(seed, 0, L, i, t, 0))
                       for i in range(n)])
        oracle.run(n, wl.star(n), x, mu, msg, counts, lr, sigma, seed, t, 1, 0)
        assert np.allclose(x[0], xh.mean(axis=0), rtol=1e-13, atol=1e-13)


@pytest.mark.parametrize("shape", ["chain", "binary", "star", "torus"])
def test_converges_to_mean_of_centres_without_noise(shape):
    """sigma = 0: the unique fixed point is x_i = mean_j mu_j on every tree,
    reached linearly whatever the heterogeneity (appendix "Independence of
    heterogeneity")."""
    n = 16 if shape == "torus" else 12
    edges = {"chain": wl.chain(n), "binary": wl.binary_tree(n), "star": wl.star(n),
             "torus": wl.torus_spanning_tree(4, 4, 1)}[shape]
    L = 6
    rng = np.random.default_rng(4)
    mu = 5.0 * rng.normal(size=(n, L))
    x = np.zeros((n, L))
    E = 2 * (n - 1)
    oracle.run(n, edges, x, mu, np.zeros((E, L)), np.zeros(E, np.int32), 0.3, 0.0, 0, 0, 600, 1)
    assert np.max(np.abs(x - mu.mean(axis=0))) < 1e-9


# --------------------------------------------------- objective and x^0 fills

def test_mu_identity_mix_is_scaled_normals():
    n, L = 5, 4000
    mu = oracle.fill_mu(n, np.eye(n), 2.0, 9, 0, L)
    for i in range(n):
        assert np.array_equal(mu[i], 2.0 * oracle.normals(9, 0, L, row=i, step=0, stream=1))
        assert abs(mu[i].std() - 2.0) < 0.1


def test_mu_is_linear_in_the_mixture():
    """mu(mix) = mix @ [N_0; ...; N_{K-1}]: catches a transposed mixture index."""
    n, K, L = 4, 3, 50
    mix = np.random.default_rng(5).dirichlet(np.ones(K), size=n)
    centres = oracle.fill_mu(K, np.eye(K), 1.0, 2, 8, L)
    mu = oracle.fill_mu(n, mix, 1.5, 2, 8, L)
    assert np.allclose(mu, 1.5 * mix @ centres, rtol=1e-13, atol=1e-13)


def test_x0_is_shared_by_all_workers():
    x = oracle.fill_x0(6, 0.1, 3, 100, 2000)
    assert all(np.array_equal(x[0], x[i]) for i in range(6))
    assert abs(x[0].std() - 0.1) < 0.01


def test_slices_reproduce_the_full_vector():
    """Coordinates are independent and the noise is keyed by the absolute
    coordinate: a run on a slice equals the same columns of the full run."""
    n, L = 5, 37
    edges = wl.random_tree(n, 7)
    E = 2 * (n - 1)
    mix = np.eye(n)
    full = oracle.State(n, edges, L)
    full.init(0.1, 3, mix, 1.0, 4)
    full.advance(9, 0.1, 0.2, 3, mode=1)
    part = oracle.State(n, edges, 13, c0=20)
    part.init(0.1, 3, mix, 1.0, 4)
    part.advance(9, 0.1, 0.2, 3, mode=1)
    assert np.array_equal(part.x, full.x[:, 20:33])
    assert np.array_equal(part.msg, full.msg[:, 20:33])
    assert E == part.E
