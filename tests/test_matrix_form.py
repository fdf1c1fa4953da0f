"""Pin of the oracle against the paper's matrix form of RelaySGD (Section 5 and
the definition of the mixing matrix W in the appendix).

The models and gradients of the last tau_max + 1 steps are stacked into
Y^t, G^t (row n*tau + i holds worker i at time t - tau); then
Y^{t+1} = W Y^t - gamma W~ G^t, with W's first block row putting 1/n on the
copy of worker j delayed by worker i's delay to j, identity blocks shifting
the history down, and W~ equal to W's first block row alone.  The delay
follows Algorithm 1 taken literally, max(tau_ij - 1, 0), tau_ij the hop
count; the un-shifted tau_ij that the paper's delayed-average formula
prints does not reproduce the iterates, which the last test records.

W is built here from breadth-first distances alone (no messages, no
counters), so agreement checks the oracle's message recursion, counters and
rebuild against an independent linear recurrence.
"""
import numpy as np
import pytest

from oracle import oracle
from paper_2110_04175_gb300 import workloads as wl
from tests import treeutil as tu


def mixing_matrices(n, tau, shift=1):
    """(W, W~, tau_max) for delays max(tau_ij - shift, 0)."""
    delay = np.maximum(np.asarray(tau) - shift, 0)
    tmax = int(delay.max()) if n > 1 else 0
    N = n * (tmax + 1)
    W = np.zeros((N, N))
    for i in range(n):
        for j in range(n):
            W[i, n * delay[i, j] + j] += 1.0 / n
    Wt = W.copy()
    for s in range(1, tmax + 1):
        for i in range(n):
            W[n * s + i, n * (s - 1) + i] = 1.0
    return W, Wt, tmax


def oracle_history(n, edges, L, steps, mode, lr, sigma, seed, mu, x0):
    """x^0 .. x^steps of the oracle, one step per call."""
    E = 2 * (n - 1)
    x = x0.copy()
    msg = np.zeros((E, L))
    counts = np.zeros(E, np.int32)
    hist = [x.copy()]
    for t in range(steps):
        oracle.run(n, edges, x, mu, msg, counts, lr, sigma, seed, t, 1, mode)
        hist.append(x.copy())
    return hist


def gradient(hist, mu, s, sigma, seed):
    """grad F_i(x_i^s; xi_i^s) for every worker: (x - mu) + sigma xi, xi the
    stream-0 normal of worker i at step s."""
    n, L = mu.shape
    xi = np.stack([oracle.normals(seed, 0, L, row=i, step=s, stream=0) for i in range(n)])
    return (hist[s] - mu) + sigma * xi


def matrix_form_error(n, edges, mode, shift=1, extra=8, L=5, sigma=0.3, seed=3):
    """Largest gap between the oracle and the matrix recurrence started from
    the oracle's history at t0 = diam - 1 (the first step after which every
    worker has heard from every other) and run `extra` steps on its own."""
    tau = np.asarray(tu.distances(n, edges))
    diam = int(tau.max())
    W, Wt, tmax = mixing_matrices(n, tau, shift)
    rng = np.random.default_rng(n * 31 + len(edges))
    mu = rng.normal(size=(n, L))
    x0 = np.tile(rng.normal(size=L), (n, 1))
    lr = 0.2
    t0 = max(diam - 1, tmax)
    hist = oracle_history(n, edges, L, t0 + extra, mode, lr, sigma, seed, mu, x0)
    Y = np.concatenate([hist[t0 - s] for s in range(tmax + 1)])
    worst = 0.0
    for t in range(t0, t0 + extra):
        G = np.concatenate([gradient(hist, mu, t - s, sigma, seed) for s in range(tmax + 1)])
        Y = W @ Y - lr * (Wt @ G)
        # the whole stack: the new models on top, the shifted history below
        want = np.concatenate([hist[t + 1 - s] for s in range(tmax + 1)])
        worst = max(worst, float(np.max(np.abs(Y - want))))
    return worst


def _trees():
    out = [(n, e) for n in (2, 3, 4, 5) for e in tu.all_trees(n)]
    out += [(8, wl.chain(8)), (10, wl.binary_tree(10)), (7, wl.star(7)),
            (9, wl.torus_spanning_tree(3, 3, 0)), (9, wl.random_tree(9, 2))]
    return out


TREES = _trees()


@pytest.mark.parametrize("mode", [0, 1])
def test_oracle_follows_the_matrix_form_after_warm_up(mode):
    """Every tree on up to 5 nodes and a few larger ones: the matrix
    recurrence, seeded with the oracle's history, reproduces the oracle's
    next iterates to rounding (both rebuild rules coincide once nbar = n)."""
    for n, edges in TREES:
        err = matrix_form_error(n, np.asarray(edges, np.int32).reshape(-1, 2), mode)
        assert err < 1e-12, (n, edges, err)


def test_mixing_matrix_is_row_stochastic_with_the_stated_blocks():
    """W 1 = 1, W >= 0; the first block row sums to (1/n) 1 1^T over its
    blocks; spectral radius 1, with W^k converging to 1 pi^T for the left
    Perron vector pi (the augmented graph has self-loops, so it is
    aperiodic)."""
    for n, edges in TREES:
        if n == 1:
            continue
        tau = np.asarray(tu.distances(n, np.asarray(edges).reshape(-1, 2)))
        W, Wt, tmax = mixing_matrices(n, tau)
        N = W.shape[0]
        assert np.all(W >= 0)
        assert np.allclose(W @ np.ones(N), 1.0, rtol=0, atol=1e-15)
        blocks = sum(W[:n, n * s:n * (s + 1)] for s in range(tmax + 1))
        assert np.allclose(blocks, np.full((n, n), 1.0 / n), rtol=0, atol=1e-15)
        assert np.array_equal(Wt[n:], np.zeros((N - n, N)))
        assert np.array_equal(Wt[:n], W[:n])
        ev, vl = np.linalg.eig(W.T)
        k = int(np.argmax(np.abs(ev)))
        assert abs(ev[k] - 1.0) < 1e-10
        pi = np.real(vl[:, k])
        pi = pi / pi.sum()
        assert np.all(pi >= -1e-12)
        Wk = np.linalg.matrix_power(W, 400)
        assert np.max(np.abs(Wk - np.outer(np.ones(N), pi))) < 1e-8


def test_unshifted_delays_do_not_reproduce_the_iterates():
    """With delays tau_ij (not tau_ij - 1) the recurrence misses the oracle
    on every tree with more than two nodes: Algorithm 1 read literally
    hears a worker at distance tau after tau - 1 steps."""
    for n, edges in [(3, wl.chain(3)), (8, wl.chain(8)), (7, wl.star(7)),
                     (10, wl.binary_tree(10))]:
        err = matrix_form_error(n, edges, 1, shift=0)
        assert err > 1e-3, (n, err)
