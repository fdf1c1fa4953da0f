"""Shared helpers of the GPU parity tests: run the CUDA path, run the oracle on
chosen coordinates, compare with the parity metric.

Parity metric (per array, padding excluded):
    max_e |g_e - r_e| / max(|r_e|, rms(r))  <=  1e-5
with g the fp32 GPU value and r the fp64 oracle value; counters must be equal.
parity_report adds the plain errors beside it (max absolute, max relative,
and how many elements sit below the rms floor); the full-size tests record
them when RELAY_PARITY_LOG names a file.
The fp32 path differs from the fp64 definition only by rounding: a float32
restatement of the step stays within 1e-6 of the oracle on every workload
(10x below the bar), so 1e-5 leaves room for the GPU's own summation order
and its fp32 normals (within NORMAL_ABS_ERR of the oracle's).
"""
from __future__ import annotations

import os

import numpy as np
import torch

import paper_2110_04175_gb300 as rs
from oracle import oracle

RTOL = 1e-5

# How far a normal drawn on the GPU can sit from the oracle's fp64 Box-Muller
# of the same Philox uniforms.  The GPU forms z = r (cos, sin)(theta) with
# r = sqrt(-2 ln u), u >= 2^-24 (so r <= sqrt(48 ln 2) = 5.77), using CUDA's
# logf, sqrt.approx and the fast __sincosf on theta = 2 pi u - pi, computed
# with one fp32 fma.  Terms, at r = 5.77:
#   theta's error: |pi_f - pi| + half an ulp at |theta| <= pi, 3.3e-7, times r     1.9e-6
#   __sincosf: at most 2^-21.41 absolute on [-pi, pi] (CUDA's stated bound), times r 2.1e-6
#   r: logf (1 ulp) and sqrt.approx (taken as 2^-22 relative), times |z|            1.6e-6
#   the product's rounding, 2^-24 |z|                                               0.4e-6
# test_normal_generator_error_within_derived_bound measures it on 8.4M normals
# (largest deviation 1.6e-6).
NORMAL_ABS_ERR = 6e-6

# When set, the full-size parity tests append one JSON line per compared
# array to this file: the metric above and the plain errors beside it.
PARITY_LOG = os.environ.get("RELAY_PARITY_LOG")


def parity_error(g: np.ndarray, r: np.ndarray) -> float:
    g = np.asarray(g, dtype=np.float64)
    r = np.asarray(r, dtype=np.float64)
    if r.size == 0:
        return 0.0
    rms = float(np.sqrt(np.mean(r * r)))
    denom = np.maximum(np.abs(r), rms if rms > 0 else 1.0)
    return float(np.max(np.abs(g - r) / denom))


def parity_report(g: np.ndarray, r: np.ndarray) -> dict:
    """The parity metric with the plain errors beside it:
    floored        max |g - r| / max(|r|, rms(r)) (the bar, 1e-5);
    abs_max        max |g - r|;
    rel_max        max |g - r| / |r| over the elements with r != 0;
    rel_max_at     |r| / rms(r) at that element (how close to zero it sits);
    rel_max_big    max |g - r| / |r| over the elements with |r| >= rms(r),
                   where the two metrics coincide;
    floor_share    the fraction of elements whose denominator is the rms
                   floor (|r| < rms(r)) rather than |r|;
    over_bar_share the fraction whose plain relative error exceeds 1e-5."""
    g = np.asarray(g, dtype=np.float64).ravel()
    r = np.asarray(r, dtype=np.float64).ravel()
    out = {"elements": int(r.size)}
    if r.size == 0:
        return out
    diff = np.abs(g - r)
    rms = float(np.sqrt(np.mean(r * r)))
    a = np.abs(r)
    out["rms"] = rms
    out["floored"] = float(np.max(diff / np.maximum(a, rms if rms > 0 else 1.0)))
    out["abs_max"] = float(diff.max())
    nz = a > 0
    if nz.any():
        rel = diff[nz] / a[nz]
        k = int(np.argmax(rel))
        out["rel_max"] = float(rel[k])
        out["rel_max_at"] = float(a[nz][k] / rms) if rms > 0 else None
        out["over_bar_share"] = float(np.mean(rel > RTOL)) * float(nz.mean())
    big = a >= rms
    out["rel_max_big"] = float(np.max(diff[big] / a[big])) if big.any() else None
    out["floor_share"] = float(np.mean(a < rms))
    return out


def generated_input_error(mix, mu_scale: float, sigma: float, x0_std: float) -> np.ndarray:
    """Per worker ([n][1]), how far the gradient's generated inputs may sit
    from the oracle's: mu_i = mu_scale sum_k mix_ik N_k, sigma xi_i and the
    shared x^0 = x0_std N are normals, each within NORMAL_ABS_ERR."""
    mix = np.abs(np.asarray(mix, dtype=np.float64))
    return ((mu_scale * mix.sum(axis=1) + sigma + x0_std) * NORMAL_ABS_ERR)[:, None]


def record_parity(label: str, array: str, g, r):
    """Appends parity_report(g, r) for `array` of case `label` to PARITY_LOG (if set)."""
    if not PARITY_LOG:
        return
    import json
    with open(PARITY_LOG, "a") as f:
        f.write(json.dumps({"case": label, "array": array, **parity_report(g, r)}) + "\n")


def gpu_run(w, steps: int, mode: int | None = None, d: int | None = None, c0: int = 0,
            stream=None, objective: str = "generated", kernel: str = "auto") -> rs.RelayRun:
    """Runs `steps` RelaySGD steps of workload `w` on cuda:0 through the C ABI."""
    run = rs.RelayRun(w.n, w.d if d is None else d, w.edges, device="cuda:0",
                      mode=w.mode if mode is None else mode, c0=c0, objective=objective,
                      kernel=kernel)
    run.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
    for _ in range(steps):
        run.step(w.lr, w.seed, stream)
    torch.cuda.synchronize()
    return run


def oracle_range(w, c0: int, length: int, steps: int, mode: int | None = None) -> oracle.State:
    st = oracle.State(w.n, w.edges, length, c0=c0)
    st.init(w.x0_std, w.seed, w.mix.astype(np.float64), w.mu_scale, w.mu_seed)
    st.advance(steps, float(np.float32(w.lr)), float(np.float32(w.sigma)), w.seed,
               w.mode if mode is None else mode)
    return st


def windows(d: int, width: int = 16384):
    """Every coordinate of [0, d) as consecutive windows (parallel oracle work)."""
    return [(s, min(width, d - s)) for s in range(0, d, width)]


def c8_sample(d: int, seed: int, edge: int = 65536, n_windows: int = 1024, width: int = 1024):
    """The full-size parity sample: the first and the last `edge` coordinates
    (the last quad's ragged tail included) and `n_windows` random windows of
    `width` coordinates between them (about a million coordinates)."""
    if d <= 2 * edge + width:
        return windows(d)
    rng = np.random.default_rng(seed)
    blocks = (d - 2 * edge) // width
    picks = np.sort(rng.choice(blocks, size=min(n_windows, blocks), replace=False))
    return ([(0, edge)] + [(edge + int(b) * width, width) for b in picks] + [(d - edge, edge)])


def sample_columns(d: int, head: int, tail: int, n_random: int, seed: int = 0):
    """Contiguous ranges (start, length) to compare: the first `head`
    coordinates, the last `tail` (ragged end of the last quad included) and
    `n_random` single coordinates drawn uniformly."""
    rng = np.random.default_rng(seed)
    ranges = [(0, min(head, d))]
    if d > head:
        start = max(head, d - tail)
        ranges.append((start, d - start))
    for c in rng.choice(np.arange(head, max(head + 1, d - tail)), size=min(n_random, max(0, d - head - tail)),
                        replace=False):
        ranges.append((int(c), 1))
    return ranges


def parallel_map(fn, items) -> list:
    """fn over items on the host cores, in order: for oracle work, whose ctypes
    calls release the GIL and which keeps no shared state."""
    from concurrent.futures import ThreadPoolExecutor
    items = list(items)
    threads = max(1, min(len(items), len(os.sched_getaffinity(0))))
    with ThreadPoolExecutor(threads) as pool:
        return list(pool.map(fn, items))


def oracle_ranges(w, ranges, steps: int, mode: int | None = None, c0: int = 0) -> list:
    """oracle_range for every (start, length) window, run concurrently."""
    return parallel_map(lambda r: oracle_range(w, c0 + r[0], r[1], steps, mode), ranges)


def compare_ranges(run: rs.RelayRun, w, ranges, steps: int, mode: int | None = None, c0: int = 0,
                   label: str | None = None):
    """Max parity error of x and of the last messages over the given ranges;
    asserts the counters are bit-exact.  With a label, the plain errors are
    recorded too (record_parity)."""
    gx, gm, ox, om = [], [], [], []
    counts = None
    for (start, length), st in zip(ranges, oracle_ranges(w, ranges, steps, mode, c0)):
        gx.append(run.x[:, start:start + length].double().cpu().numpy())
        gm.append(run.messages[:run.E, start:start + length].double().cpu().numpy())
        ox.append(st.x)
        om.append(st.msg)
        counts = st.counts
    g_counts = run.counts[:run.E].cpu().numpy()
    assert np.array_equal(g_counts, counts), (g_counts, counts)
    gx, ox = np.concatenate(gx, axis=1), np.concatenate(ox, axis=1)
    ex = parity_error(gx, ox)
    em = 0.0
    if run.E:
        gm, om = np.concatenate(gm, axis=1), np.concatenate(om, axis=1)
        em = parity_error(gm, om)
    if label:
        record_parity(label, "x", gx, ox)
        if run.E:
            record_parity(label, "messages", gm, om)
    return ex, em


def adam_step_bound(x, mu, xi, sigma: float, m, v, lr: float, beta1: float, beta2: float, eps: float,
                    t: int, dnoise=0.0) -> np.ndarray:
    """Per coordinate, how far fp32 rounding can move one Adam step (t from
    0) of any worker, from the oracle's state before the step (x, mu, the
    noise xi) and after it (first and second moments m, v), all [n][len].

    Adam divides by sqrt(v_hat) + eps, so a rounding error dg in a gradient
    moves the update by lr (1 - beta1) / (1 - beta1^k) dg / (sqrt(v_hat) +
    eps): large wherever a worker's gradient is small against its history.
    The update's own rounding (8 ulp of |u|) adds up too, since |u| stays
    near lr however small the gradient.  At the first step the update is
    -lr g / (|g| + eps), in effect -lr sign(g) when eps is tiny: within
    rounding of zero the sign is a decision that two precisions may take
    differently, a difference of 2 lr.  dg is the fp32 rounding of the
    gradient's terms, 2^-23 (|x| + |mu| + sigma |xi|), plus `dnoise`, how far
    the generated inputs of the gradient (the centres, the noise and the
    initial model, drawn as normals) may sit from the oracle's:
    (mu_scale sum_k |mix_ik| + sigma + x0_std) NORMAL_ABS_ERR per worker
    ([n][1], or a scalar).  The relay and rebuild only average, so the
    largest worker's value bounds the step's effect on every worker; summed
    over steps it bounds the trajectory."""
    g = (x - mu) + sigma * xi
    dg = 2.0 ** -23 * (np.abs(x) + np.abs(mu) + sigma * np.abs(xi)) + dnoise
    k = t + 1
    denom = np.sqrt(v / (1.0 - beta2 ** k)) + eps
    du = lr * (1.0 - beta1) / (1.0 - beta1 ** k) * dg / denom
    if t == 0:
        du = np.where(np.abs(g) <= 4.0 * dg, 2.0 * lr, du)
    du = du + 8.0 * 2.0 ** -24 * (lr / (1.0 - beta1 ** k) * np.abs(m) / denom)
    return du.max(axis=0)

