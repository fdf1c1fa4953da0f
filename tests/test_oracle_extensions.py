"""Pins of the oracle's extensions: local momentum / Adam (appendix "RelaySGD
with momentum", "RelaySGD with Adam") and lost messages with the robust
rebuild (Section 4.4, Table 5).

- The local optimisers are checked against PyTorch's own SGD(nesterov) and
  Adam in float64 on one worker (the paper uses "the standard Adam
  implementation of PyTorch"), and on two workers, where RelaySGD is exact
  all-reduce averaging of the workers' locally-updated models.
- Lost messages are checked against an exact-rational routing brute force:
  a model reaches a worker iff every hop of its path was delivered at the
  step the hop happened.
"""
from fractions import Fraction

import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2110_04175_gb300 import workloads as wl
from tests import treeutil as tu


def _grad_noise(seed, c0, L, row, step):
    return oracle.normals(seed, c0, L, row=row, step=step, stream=0)


# ---------------------------------------------------------- local optimisers

def test_nesterov_with_zero_momentum_is_sgd():
    n, L = 7, 9
    edges = wl.random_tree(n, 1)
    rng = np.random.default_rng(0)
    mu = rng.normal(size=(n, L))
    a = oracle.State(n, edges, L)
    b = oracle.State(n, edges, L)
    for st in (a, b):
        st.x = np.tile(rng.normal(size=L), (n, 1)) if st is a else a.x.copy()
        st.mu = mu.copy()
    a.advance(12, 0.2, 0.3, 5, mode=1)
    b.advance(12, 0.2, 0.3, 5, mode=1, opt=oracle.OPT_NESTEROV, beta1=0.0)
    assert np.array_equal(a.x, b.x) and np.array_equal(a.msg, b.msg)


def _torch_single_worker(kind, x0, mu, lr, sigma, seed, steps, **kw):
    p = torch.nn.Parameter(torch.tensor(x0, dtype=torch.float64))
    if kind == "nesterov":
        opt = torch.optim.SGD([p], lr=lr, momentum=kw["beta1"], nesterov=True)
    else:
        opt = torch.optim.Adam([p], lr=lr, betas=(kw["beta1"], kw["beta2"]), eps=kw["eps"])
    for t in range(steps):
        xi = torch.tensor(_grad_noise(seed, 0, len(x0), 0, t))
        opt.zero_grad()
        p.grad = (p.detach() - torch.tensor(mu)) + sigma * xi
        opt.step()
    return p.detach().numpy()


@pytest.mark.parametrize("kind", ["nesterov", "adam"])
def test_single_worker_matches_pytorch_optimizer(kind):
    L, steps = 16, 30
    rng = np.random.default_rng(1)
    mu = rng.normal(size=L) * 2
    x0 = rng.normal(size=L)
    kw = dict(beta1=0.9, beta2=0.99, eps=1e-8)
    want = _torch_single_worker(kind, x0, mu, 0.05, 0.1, 7, steps, **kw)
    st = oracle.State(1, np.zeros((0, 2), np.int32), L)
    st.x = x0[None, :].copy()
    st.mu = mu[None, :].copy()
    opt = oracle.OPT_NESTEROV if kind == "nesterov" else oracle.OPT_ADAM
    st.advance(steps, 0.05, 0.1, 7, mode=0, opt=opt, **kw)
    assert np.allclose(st.x[0], want, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("kind", ["nesterov", "adam"])
def test_two_workers_average_locally_updated_models(kind):
    """n = 2: after every step both workers hold the mean of their two local
    optimiser steps (each worker keeps its own optimiser state)."""
    L, steps = 8, 12
    rng = np.random.default_rng(2)
    mu = rng.normal(size=(2, L))
    x0 = rng.normal(size=L)
    kw = dict(beta1=0.8, beta2=0.95, eps=1e-6)
    params = [torch.nn.Parameter(torch.tensor(x0)) for _ in range(2)]
    if kind == "nesterov":
        opts = [torch.optim.SGD([p], lr=0.1, momentum=kw["beta1"], nesterov=True) for p in params]
    else:
        opts = [torch.optim.Adam([p], lr=0.1, betas=(kw["beta1"], kw["beta2"]), eps=kw["eps"])
                for p in params]
    st = oracle.State(2, [(0, 1)], L)
    st.x = np.tile(x0, (2, 1))
    st.mu = mu.copy()
    opt = oracle.OPT_NESTEROV if kind == "nesterov" else oracle.OPT_ADAM
    for t in range(steps):
        for i in range(2):
            xi = torch.tensor(_grad_noise(3, 0, L, i, t))
            opts[i].zero_grad()
            params[i].grad = (params[i].detach() - torch.tensor(mu[i])) + 0.2 * xi
            opts[i].step()
        avg = (params[0].detach() + params[1].detach()) / 2
        with torch.no_grad():
            for p in params:
                p.copy_(avg)
        st.advance(1, 0.1, 0.2, 3, mode=0, opt=opt, **kw)
        assert np.allclose(st.x, np.tile(avg.numpy(), (2, 1)), rtol=1e-12, atol=1e-12)


# -------------------------------------------------------------- lost messages

@pytest.mark.parametrize("mode", [0, 1])
def test_all_messages_lost_isolates_the_workers(mode):
    """Nothing arrives: nbar = 1, so mode 0 keeps x^{t+1/2} and mode 1 gives
    (x^{t+1/2} + (n - 1) x^t) / n; every message and counter reads 0."""
    n, L = 6, 5
    edges = wl.random_tree(n, 2)
    rng = np.random.default_rng(4)
    mu = rng.normal(size=(n, L))
    x = rng.normal(size=(n, L))
    st = oracle.State(n, edges, L)
    st.x, st.mu = x.copy(), mu.copy()
    for t in range(4):
        xh = np.array([x[i] - 0.3 * ((x[i] - mu[i]) + 0.1 * _grad_noise(9, 0, L, i, t))
                       for i in range(n)])
        x = xh if mode == 0 else (xh + (n - 1) * x) / n
        nbar = st.advance(1, 0.3, 0.1, 9, mode=mode, drop=np.ones((1, 2 * (n - 1))))
        assert np.allclose(st.x, x, rtol=1e-13, atol=1e-13)
        assert np.all(st.msg == 0) and np.all(st.counts == 0) and np.all(nbar == 1)


def _routing_with_losses(n, edges, x0, mu, lr, steps, mode, lost):
    """Exact routing view with lost messages: x_l^{(s)+1/2} reaches i at step
    s + tau - 1 iff each hop p_h -> p_{h+1} of the path l -> i was delivered at
    step s + h.  Returns per-step models and counters (count of models behind
    each directed edge's message)."""
    tau = tu.distances(n, edges)
    adj = tu.adjacency(n, edges)
    dedges = tu.directed(edges)
    eid = {e: k for k, e in enumerate(dedges)}

    def path(a, b):  # nodes from a to b
        prev = {a: None}
        q = [a]
        for u in q:
            for v in adj[u]:
                if v not in prev:
                    prev[v] = u
                    q.append(v)
        p = [b]
        while p[-1] != a:
            p.append(prev[p[-1]])
        return p[::-1]

    paths = {(a, b): path(a, b) for a in range(n) for b in range(n)}

    def arrives(l, i, s):  # x_l^{(s)+1/2} along l -> i, hop h at step s + h
        p = paths[(l, i)]
        return all(not lost[s + h][eid[(p[h], p[h + 1])]] for h in range(len(p) - 1))

    L = len(x0[0])
    xs, xhs, counts = [x0], [], []
    for t in range(steps):
        xt = xs[t]
        xhs.append([[xt[i][c] - lr * (xt[i][c] - mu[i][c]) for c in range(L)] for i in range(n)])
        nxt = []
        for i in range(n):
            B = [l for l in range(n) if tau[i][l] <= t + 1 and
                 (l == i or arrives(l, i, t - tau[i][l] + 1))]
            row = []
            for c in range(L):
                s = sum(xhs[t - max(tau[i][l] - 1, 0)][l][c] for l in B)
                row.append(s / len(B) if mode == 0 else (s + (n - len(B)) * xt[i][c]) / n)
            nxt.append(row)
        xs.append(nxt)
        # counter of edge a -> b at step t: models of T_{a\b} that reached a in
        # time and whose last hop a -> b at step t was delivered
        cnt = []
        for (a, b) in dedges:
            side = tu.side(n, edges, a, b)
            k = 0
            if not lost[t][eid[(a, b)]]:
                for l in side:
                    s = t - tau[a][l]
                    if s >= 0 and (l == a or arrives(l, a, s)):
                        k += 1
            cnt.append(k)
        counts.append(cnt)
    return xs, counts


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("n", [2, 3, 4, 5])
def test_lost_messages_equal_routing_brute_force(n, mode):
    rng = np.random.default_rng(10 * n + mode)
    trees = list(tu.all_trees(n))
    if len(trees) > 25:
        trees = [trees[k] for k in rng.choice(len(trees), 25, replace=False)]
    lr = Fraction(1, 4)
    L = 2
    for edges in trees:
        E = 2 * len(edges)
        steps = tu.diameter(n, edges) + 4
        lost = (rng.random((steps, E)) < 0.3).astype(np.uint8)
        x0i = rng.integers(-9, 9, size=(n, L))
        mui = rng.integers(-9, 9, size=(n, L))
        xs, cnts = _routing_with_losses(n, edges, [[Fraction(int(v)) for v in r] for r in x0i],
                                        [[Fraction(int(v)) for v in r] for r in mui], lr, steps,
                                        mode, lost)
        st = oracle.State(n, edges, L)
        st.x, st.mu = x0i.astype(np.float64), mui.astype(np.float64)
        for t in range(steps):
            st.advance(1, float(lr), 0.0, 0, mode=mode, drop=lost[t:t + 1])
            exact = np.array([[float(v) for v in r] for r in xs[t + 1]])
            assert np.max(np.abs(st.x - exact)) <= 1e-12 * max(1.0, np.max(np.abs(exact)))
            assert list(st.counts) == cnts[t], (edges, t)


# ------------------------------------------------ RelaySum/Grad and DME

def _delays(n, edges):
    tau = tu.distances(n, edges)
    return [[max(tau[i][l] - 1, 0) for l in range(n)] for i in range(n)]


@pytest.mark.parametrize("n", [1, 2, 3, 4, 5, 6])
def test_relaysum_grad_equals_delayed_update_sums(n):
    """Algorithm 6: every update u_l^s = -lr grad reaches every worker i, with
    weight exactly 1/n, at step s + max(tau_il - 1, 0):
        x_i^{t+1} = x_i^0 + 1/n sum_l sum_{s <= t - delta_il} u_l^s."""
    rng = np.random.default_rng(50 + n)
    trees = list(tu.all_trees(n))
    if len(trees) > 30:
        trees = [trees[k] for k in rng.choice(len(trees), 30, replace=False)]
    lr = Fraction(1, 4)
    L = 2
    for edges in trees:
        delta = _delays(n, edges)
        steps = tu.diameter(n, edges) + 3
        x0i = rng.integers(-9, 9, size=(n, L))
        mui = rng.integers(-9, 9, size=(n, L))
        xs = [[[Fraction(int(v)) for v in r] for r in x0i]]
        us = []
        for t in range(steps):
            us.append([[-lr * (xs[t][l][c] - mui[l][c]) for c in range(L)] for l in range(n)])
            xs.append([[xs[0][i][c] + sum(us[s][l][c] for l in range(n)
                                          for s in range(0, t - delta[i][l] + 1)) / n
                        for c in range(L)] for i in range(n)])
        st = oracle.State(n, edges, L)
        st.x, st.mu = x0i.astype(np.float64), mui.astype(np.float64)
        for t in range(steps):
            st.advance(1, float(lr), 0.0, 0, algo=oracle.ALGO_GRAD)
            exact = np.array([[float(v) for v in r] for r in xs[t + 1]])
            assert np.max(np.abs(st.x - exact)) <= 1e-12 * max(1.0, np.max(np.abs(exact))), edges


@pytest.mark.parametrize("n", [1, 2, 3, 4, 5, 6])
def test_dme_equals_delayed_sample_sums(n):
    """Algorithm 5: y_i^{t+1} = sum_l sum_{s <= t - delta_il} dhat_l^s and
    s_i^{t+1} counts those samples."""
    rng = np.random.default_rng(60 + n)
    trees = list(tu.all_trees(n))
    if len(trees) > 30:
        trees = [trees[k] for k in rng.choice(len(trees), 30, replace=False)]
    L, sigma, seed = 3, 0.5, 21
    for edges in trees:
        delta = _delays(n, edges)
        steps = tu.diameter(n, edges) + 3
        mui = rng.integers(-5, 5, size=(n, L)).astype(np.float64)
        samples = [[[Fraction(float(mui[l][c] + sigma * oracle.normal(seed, c, l, s, 0)))
                     for c in range(L)] for l in range(n)] for s in range(steps)]
        st = oracle.State(n, edges, L)
        st.x, st.mu = np.zeros((n, L)), mui.copy()
        for t in range(steps):
            st.advance(1, 0.0, sigma, seed, algo=oracle.ALGO_DME)
            y = np.array([[float(sum(samples[s][l][c] for l in range(n)
                                     for s in range(0, t - delta[i][l] + 1))) for c in range(L)]
                          for i in range(n)])
            cnt = [sum(max(t - delta[i][l] + 1, 0) for l in range(n)) for i in range(n)]
            assert np.allclose(st.x, y, rtol=1e-12, atol=1e-12), edges
            assert list(st.dme_count) == cnt


def test_dme_variance_shrinks_like_one_over_samples():
    """With i.i.d. N(1, sigma^2) samples, worker i's estimate y_i / s_i has
    variance sigma^2 / s_i (appendix: variance reduction O(1/(nT)))."""
    n, L, sigma, steps = 8, 20000, 1.0, 12
    st = oracle.State(n, wl.binary_tree(n), L)
    st.x, st.mu = np.zeros((n, L)), np.ones((n, L))
    st.advance(steps, 0.0, sigma, 4, algo=oracle.ALGO_DME)
    for i in range(n):
        est = st.x[i] / st.dme_count[i]
        assert abs(est.mean() - 1.0) < 5 * sigma / np.sqrt(st.dme_count[i] * L)
        assert abs(est.var() * st.dme_count[i] / sigma ** 2 - 1.0) < 0.05


# ------------------------------------------------ learning-rate correction

def _alpha(n, edges, mode, steps=3000):
    E = 2 * (n - 1)
    x = np.zeros((n, 1))
    mu = np.ones((n, 1))
    msg = np.zeros((E, 1))
    c = np.zeros(E, np.int32)
    oracle.run(n, edges, x, mu, msg, c, 1.0, 0.0, 0, 0, 1, mode)
    oracle.run(n, edges, x, mu, msg, c, 0.0, 0.0, 0, 1, steps, mode)
    return x[:, 0]


def test_lr_correction_closed_forms():
    """Algorithm 1's division by nbar loses nothing (alpha = 1 on any tree);
    so does any rule on n <= 2 (all-reduce from the first step).  Under the
    robust rule alpha < 1 and is the same on every worker."""
    for edges in (wl.chain(9), wl.binary_tree(11), wl.star(7), wl.random_tree(12, 3)):
        n = int(np.max(edges)) + 1
        assert np.allclose(_alpha(n, edges, 0), 1.0, rtol=0, atol=1e-12)
        a = _alpha(n, edges, 1)
        assert 0.0 < a.mean() < 1.0 and np.ptp(a) < 1e-9
    assert np.allclose(_alpha(2, [(0, 1)], 1), 1.0, atol=1e-12)
    assert np.allclose(_alpha(1, np.zeros((0, 2), np.int32), 1), 1.0, atol=1e-12)
