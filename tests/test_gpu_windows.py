"""relay_step_windows: the tree windows of the double binary trees (Section 3,
"Spanning trees") stepped by one counter launch and one step-kernel launch.

Each case runs the same double-tree state twice -- once through
relay_step_windows, once through relay_step window by window -- and requires
the models, both windows' messages, counters, optimiser state and
mean-estimation counts to agree bit for bit after every few steps.  The cases
force the walk kernel (the one-launch path) across the objective sources, the
local optimisers, the algorithms, lost messages, odd worker counts (the
shifted second tree), ragged and tiny windows, and windows of unequal length;
others take the fallback (the node kernel, or windows that differ in their
objective).  A last case checks the one launch against two oracle runs.
"""
import gc

import numpy as np
import pytest
import torch

import paper_2110_04175_gb300 as rs
from paper_2110_04175_gb300 import build as rs_build
from paper_2110_04175_gb300 import workloads as wl
from tests.gpu_util import RTOL, oracle_range, parity_error

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    rs_build.build()
    yield
    gc.collect()
    torch.cuda.empty_cache()


OPTS = {None: None, "nesterov": ("nesterov", 0.9), "adam": ("adam", 0.9, 0.99, 1e-3)}

CASES = {
    "n16_stored": dict(n=16, d=40_001),
    "n16_generated_dirichlet": dict(n=16, d=20_003, objective="generated", K=10),
    "n15_nesterov_lost": dict(n=15, d=9_231, optimizer="nesterov", lost_p=0.2),
    "n16_adam": dict(n=16, d=5_003, optimizer="adam"),
    "n12_grad": dict(n=12, d=3_001, algorithm="grad"),
    "n16_dme_lost": dict(n=16, d=3_001, algorithm="dme", lost_p=0.1),
    "n16_alg1_rebuild": dict(n=16, d=7_777, mode=0),
    "n2_tiny": dict(n=2, d=13),
    "n3_one_quad_each": dict(n=3, d=8),
    "n64_many_ctas": dict(n=64, d=1_000_001),
    "n16_nodes_fallback": dict(n=16, d=4_099, kernel="nodes"),
}


def _make(c, seed=5):
    n = c["n"]
    trees = list(wl.double_binary_trees(n))
    run = rs.RelayRun(n, c["d"], trees, device="cuda:0", mode=c.get("mode", 1),
                      objective=c.get("objective", "stored"), optimizer=OPTS[c.get("optimizer")],
                      algorithm=c.get("algorithm", "relaysgd"), kernel=c.get("kernel", "walk"))
    mix = wl.dirichlet_mix(n, c["K"], 0.1, seed) if "K" in c else wl.identity_mix(n)
    run.init(0.1, seed, mix, 1.0, seed + 1, 0.1)
    if c.get("algorithm") == "dme":
        run.x.zero_()
    return run


def _state(run):
    out = [run.x[:, :run.d].clone()] + [s[:, :run.d].clone() for s in run.state]
    for tr in run.trees:
        if tr.E:
            out += [tr.msg[b][:tr.E, :tr.d].clone() for b in (0, 1)] + [tr.counts.clone()]
        if tr.dme_count is not None:
            out.append(tr.dme_count.clone())
    return out


@pytest.mark.parametrize("name", sorted(CASES))
def test_step_windows_equals_relay_step_per_window(name):
    c = CASES[name]
    a, b = _make(c), _make(c)
    rng = np.random.default_rng(9)
    lr, seed = 0.05, 5
    for t in range(12):
        if c.get("lost_p"):
            for k, tr in enumerate(a.trees):
                lost = (rng.random(tr.E) < c["lost_p"]).astype(np.uint8)
                a.set_lost(lost, tree=k)
                b.set_lost(lost, tree=k)
        a.step(lr, seed)  # relay_step_windows
        for tr in b.trees:
            rs.relay_step(tr.h, b._x(tr), tr.msg[tr.cur], tr.msg[1 - tr.cur], tr.counts, lr, seed, b.t)
            tr.cur = 1 - tr.cur
        b.t += 1
        if t % 4 == 3:
            torch.cuda.synchronize()
            for u, v in zip(_state(a), _state(b)):
                assert torch.equal(u, v), (name, t)


def test_windows_with_different_objectives_fall_back():
    """Windows whose regenerated mixtures differ cannot share one launch: the
    call issues one relay_step per window, with the same results."""
    n, d = 16, 4_001
    ta, tb = wl.double_binary_trees(n)
    runs = []
    for _ in range(2):
        r = rs.RelayRun(n, d, [ta, tb], device="cuda:0", objective="generated", kernel="walk")
        r.init(0.1, 2, wl.identity_mix(n), 1.0, 3, 0.1)
        # the second window's centres from another mixture
        rs.relay_set_objective_generated(r.trees[1].h, wl.dirichlet_mix(n, 4, 0.5, 1), 4, 1.0, 3, 0.1)
        runs.append(r)
    a, b = runs
    for _ in range(6):
        a.step(0.05, 2)
        for tr in b.trees:
            rs.relay_step(tr.h, b._x(tr), tr.msg[tr.cur], tr.msg[1 - tr.cur], tr.counts, 0.05, 2, b.t)
            tr.cur = 1 - tr.cur
        b.t += 1
    torch.cuda.synchronize()
    for u, v in zip(_state(a), _state(b)):
        assert torch.equal(u, v)


def test_one_launch_windows_match_two_oracle_runs():
    n, d, steps = 16, 30_011, 20
    a, b = wl.double_binary_trees(n)
    w = wl.Workload("dbt", n, a, d, wl.identity_mix(n), 1.0, 0.05, 0.05, 0.1, steps)
    run = rs.RelayRun(n, d, [a, b], device="cuda:0", kernel="walk")
    run.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
    for _ in range(steps):
        run.step(w.lr, w.seed)
    torch.cuda.synchronize()
    for tr, edges in zip(run.trees, (a, b)):
        wt = wl.Workload("dbt", n, edges, d, w.mix, 1.0, 0.05, 0.05, 0.1, steps)
        st = oracle_range(wt, tr.col0, tr.d, steps)
        assert parity_error(run.x[:, tr.col0:tr.col0 + tr.d].double().cpu().numpy(), st.x) <= RTOL
        assert parity_error(tr.messages[:tr.E, :tr.d].double().cpu().numpy(), st.msg) <= RTOL
        assert np.array_equal(tr.counts.cpu().numpy(), st.counts)


def test_double16_full_size_one_launch_equals_forked_streams():
    """The VGG-11-sized double binary trees, 200 steps, in the launch
    configuration of the bench (stored centres, the automatic kernel: the
    walk): relay_step_windows (whose full-size parity against the oracle
    test_gpu_parity checks) equals the two windows stepped by relay_step on
    forked streams, bit for bit, where each CTA of the one launch loops over
    many quads of its window."""
    w = wl.double16_vgg11()
    states = []
    for one_launch in (True, False):
        run = rs.RelayRun(w.n, w.d, w.edges, device="cuda:0", mode=w.mode)
        run.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
        for _ in range(w.steps):
            (run.step if one_launch else run.step_forked)(w.lr, w.seed)
        torch.cuda.synchronize()
        states.append([t.cpu() for t in _state(run)])
        del run
        gc.collect()
        torch.cuda.empty_cache()
    for u, v in zip(*states):
        assert torch.equal(u, v)
