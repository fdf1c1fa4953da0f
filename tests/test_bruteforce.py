"""Exact-rational brute force of RelaySGD as delayed all-reduce averaging.

Section 3 describes RelaySGD as an all-reduce average in which worker j's
contribution reaches worker i after a delay set by their hop distance, and
notes that it could be implemented by naive peer-to-peer routing.  This test
implements that routing view directly -- no messages, no counters -- and checks
the oracle's message recursion against it on every small tree.

Reading of the delay (an ambiguity of the paper): Algorithm 1, taken line by
line, sends m^t built from m^{t-1}, receives m^t and rebuilds in the same
iteration, so worker l's half-step model reaches worker i with delay
max(tau_il - 1, 0) and the number of models received is
nbar_i^{t+1} = |{l : tau_il <= t + 1}|:

    x_i^{t+1} = 1/|B| sum_{l in B} x_l^{(t - max(tau_il - 1, 0)) + 1/2},  B = {l : tau_il <= t+1}

(the equation labelled RelaySGD prints the delay as tau_ij).  The robust
rule of Section 4.4 replaces 1/|B| by 1/n and adds (n - |B|) x_i^t.
"""
from fractions import Fraction

import numpy as np
import pytest

from oracle import oracle
from tests import treeutil as tu


def _routing_reference(n, edges, x0, mu, lr, steps, mode):
    """x^t for t = 0..steps by the routing formula, in exact rationals.

    x0, mu: lists (per worker) of lists (per coordinate) of Fractions."""
    tau = tu.distances(n, edges)
    L = len(x0[0])
    xs = [x0]        # xs[t][i][c] = x_i^t
    xhs = []         # xhs[t][i][c] = x_i^{t+1/2}
    for t in range(steps):
        xt = xs[t]
        xhs.append([[xt[i][c] - lr * (xt[i][c] - mu[i][c]) for c in range(L)] for i in range(n)])
        nxt = []
        for i in range(n):
            B = [l for l in range(n) if tau[i][l] <= t + 1]
            row = []
            for c in range(L):
                s = sum(xhs[t - max(tau[i][l] - 1, 0)][l][c] for l in B)
                if mode == 0:
                    row.append(s / len(B))
                else:
                    row.append((s + (n - len(B)) * xt[i][c]) / n)
            nxt.append(row)
        xs.append(nxt)
    return xs


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("n", [2, 3, 4, 5, 6])
def test_oracle_equals_delayed_allreduce(n, mode):
    rng = np.random.default_rng(100 * n + mode)
    trees = list(tu.all_trees(n))
    if len(trees) > 60:
        trees = [trees[k] for k in rng.choice(len(trees), 60, replace=False)]
    L = 2
    lr = Fraction(1, 4)
    for edges in trees:
        steps = tu.diameter(n, edges) + 3
        # different integer starting models per worker: the identity needs no
        # consensus at t = 0, which makes the check stronger
        x0i = rng.integers(-20, 20, size=(n, L))
        mui = rng.integers(-20, 20, size=(n, L))
        x0 = [[Fraction(int(v)) for v in row] for row in x0i]
        mu = [[Fraction(int(v)) for v in row] for row in mui]
        want = _routing_reference(n, edges, x0, mu, lr, steps, mode)
        E = 2 * len(edges)
        x = x0i.astype(np.float64)
        msg = np.zeros((E, L))
        counts = np.zeros(E, dtype=np.int32)
        for t in range(steps):
            oracle.run(n, edges, x, mui.astype(np.float64), msg, counts, float(lr), 0.0, 0, t,
                       1, mode)
            exact = np.array([[float(v) for v in row] for row in want[t + 1]])
            scale = max(1.0, float(np.max(np.abs(exact))))
            assert np.max(np.abs(x - exact)) <= 1e-12 * scale, (edges, t)
