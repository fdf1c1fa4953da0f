"""What the 1e-5 parity bar can mean for fp32 models (the parity metric's
reading of "max relative error").

Algorithm 1 computed in float32 -- any order, any hardware -- carries an
absolute rounding error of a few ulp of the values it sums (|x|, |m| of
order rms).  Where the exact result sits near zero that absolute error is
a huge relative one.  This file restates one step of Alg. 1 (robust rebuild,
Section 4.4) in plain numpy float32, in the oracle's own left-fold order, and
runs it beside the fp64 oracle on the small workloads.  It shows that:
  * the floored metric max |g - r| / max(|r|, rms(r)) of that fp32 run stays
    near 1e-6, an order of magnitude below the 1e-5 bar;
  * on the elements with |r| >= rms(r) the plain relative error is as small;
  * the plain max |g - r| / |r| over all elements exceeds 1e-5 by orders of
    magnitude, at elements within 1e-4 rms of zero: no fp32 computation of the
    step meets a plain relative bar, so the bar is read as the floored metric.
The restatement is test code only: it shares nothing with the CUDA path and
takes the noise and centres from the oracle (cast to float32) as inputs.
"""
import numpy as np
import pytest

from oracle import oracle
from paper_2110_04175_gb300 import workloads as wl

RTOL = 1e-5


def fp32_run(w, d: int, steps: int):
    """Alg. 1 (robust rebuild when w.mode == 1) in float32 over d coordinates."""
    n = w.n
    src, dst = oracle.edges(n, w.edges)
    E = len(src)
    nbr_in = [[e for e in range(E) if dst[e] == i] for i in range(n)]  # incoming edges of i
    f = np.float32
    x = oracle.fill_x0(n, w.x0_std, w.seed, 0, d).astype(f)
    mu = oracle.fill_mu(n, w.mix, w.mu_scale, w.mu_seed, 0, d).astype(f)
    msg = np.zeros((E, d), dtype=f)
    counts = np.zeros(E, dtype=np.int64)
    lr, sigma = f(w.lr), f(w.sigma)
    for t in range(steps):
        # counters and models received (integers: exact)
        c_new = np.array([1 + sum(counts[k] for k in nbr_in[src[e]] if src[k] != dst[e])
                          for e in range(E)], dtype=np.int64)
        counts = c_new
        nbar = [1 + sum(counts[k] for k in nbr_in[i]) for i in range(n)]
        # local step
        xi = np.stack([oracle.normals(w.seed, 0, d, i, t, 0) for i in range(n)]).astype(f)
        g = (x - mu) + sigma * xi
        xh = x - lr * g
        # messages: left fold in the oracle's neighbour order
        m_new = np.empty_like(msg)
        for e in range(E):
            s = xh[src[e]].copy()
            for k in nbr_in[src[e]]:
                if src[k] != dst[e]:
                    s = s + msg[k]
            m_new[e] = s
        # rebuild
        x_new = np.empty_like(x)
        for i in range(n):
            s = xh[i].copy()
            for k in nbr_in[i]:
                s = s + m_new[k]
            if w.mode == 0:
                x_new[i] = s / f(nbar[i])
            else:
                x_new[i] = (s + f(n - nbar[i]) * x[i]) / f(n)
        x, msg = x_new, m_new
    return x, msg


def oracle_run(w, d: int, steps: int):
    st = oracle.State(w.n, w.edges, d)
    st.init(w.x0_std, w.seed, w.mix.astype(np.float64), w.mu_scale, w.mu_seed)
    st.advance(steps, w.lr, w.sigma, w.seed, w.mode)
    return st.x, st.msg


def metrics(g, r):
    g = g.astype(np.float64).ravel()
    r = r.ravel()
    diff = np.abs(g - r)
    rms = float(np.sqrt(np.mean(r * r)))
    a = np.abs(r)
    floored = float(np.max(diff / np.maximum(a, rms)))
    nz = a > 0
    rel = diff[nz] / a[nz]
    k = int(np.argmax(rel))
    big = a >= rms
    return {"floored": floored, "rel_max": float(rel[k]), "rel_max_at": float(a[nz][k] / rms),
            "rel_big": float(np.max(diff[big] / a[big])), "floor_share": float(np.mean(a < rms))}


CASES = [("chain8_d4096", 4096, 100), ("binary16_d272474", 2048, 60),
         ("chain16_d9231114_dirichlet", 2048, 60), ("star64_d25000000", 512, 20)]


@pytest.mark.parametrize("name,d,steps", CASES)
def test_fp32_restatement_meets_floored_bar_not_plain_relative(name, d, steps):
    w = wl.by_name(name)
    gx, gm = fp32_run(w, d, steps)
    rx, rm = oracle_run(w, d, steps)
    for g, r in ((gx, rx), (gm, rm)):
        m = metrics(g, r)
        assert m["floored"] <= 0.3 * RTOL, m      # the bar leaves room for another fp32 order
        assert m["rel_big"] <= 0.3 * RTOL, m      # where |r| >= rms the two metrics coincide
        assert m["rel_max"] > RTOL, m             # no fp32 run meets a plain relative bar ...
        assert m["rel_max_at"] < 1e-2, m          # ... because of elements next to zero
        assert 0.6 < m["floor_share"] < 0.8, m    # ~68 %: |r| < rms for normal-like values
