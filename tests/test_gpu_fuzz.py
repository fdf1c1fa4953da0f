"""Seeded random configurations of the whole library against the oracle.

Each case draws a tree (random, star, chain or binary; up to 100 workers), a
vector length with a ragged tail, a coordinate offset, the rebuild rule, the
centre source and mixture, the local optimiser, the algorithm, a rate of lost
messages, the step kernel and whether the message buffers carry the wide
nodes' received sums, then compares every coordinate of the models
and messages, the counters (bit-exact) and the mean-estimation counts with
the oracle.  Adam cases hold every element to the 1e-5 bar plus the fp32
rounding bound derived from Adam's arithmetic (gpu_util.adam_step_bound,
with the generated inputs' error gpu_util.generated_input_error, summed over
the steps; n times that for messages): Adam's update is about lr
whatever the gradient, so its own rounding accumulates with lr, the steps and,
in messages, the workers summed.  They draw eps = 1e-2, which keeps the first
step from being a sign decision (that case is the full-size Adam test's).
"""
import gc

import numpy as np
import pytest
import torch

import paper_2110_04175_gb300 as rs
from oracle import oracle
from paper_2110_04175_gb300 import build as rs_build
from paper_2110_04175_gb300 import workloads as wl
from tests.gpu_util import RTOL, adam_step_bound, generated_input_error, parity_error

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    rs_build.build()
    yield
    gc.collect()
    torch.cuda.empty_cache()


def draw(case: int) -> dict:
    rng = np.random.default_rng(1000 + case)
    n = int(rng.choice([1, 2, 3, 5, 8, 13, 21, 34, 64, 100], p=[.05, .1, .1, .15, .15, .15, .1, .1, .05, .05]))
    shape = rng.choice(["random", "star", "chain", "binary"])
    edges = {"random": wl.random_tree(n, case) if n > 2 else wl.chain(n), "star": wl.star(n),
             "chain": wl.chain(n), "binary": wl.binary_tree(n)}[shape]
    mixkind = rng.choice(["identity", "dirichlet", "dense"])
    if mixkind == "identity":
        mix = wl.identity_mix(n)
    elif mixkind == "dirichlet":
        mix = wl.dirichlet_mix(n, int(rng.integers(2, 12)), 0.3, case)
    else:
        mix = rng.random((n, int(rng.integers(1, 9)))).astype(np.float32)
    opt = rng.choice(["sgd", "nesterov", "adam"], p=[.5, .25, .25])
    algo = rng.choice(["relaysgd", "grad", "dme"], p=[.6, .2, .2])
    c = dict(n=n, shape=str(shape), edges=np.asarray(edges, np.int32).reshape(-1, 2),
                d=int(rng.integers(1, 3000)), c0=4 * int(rng.integers(0, 50_000)), mode=int(rng.integers(0, 2)),
                objective=str(rng.choice(["stored", "generated"])), mix=mix, mixkind=str(mixkind),
                opt=str(opt), beta1=float(rng.uniform(0.5, 0.95)), beta2=float(rng.uniform(0.9, 0.999)),
                algo=str(algo), lost_p=float(rng.choice([0.0, 0.1, 0.3])),
                kernel=str(rng.choice(["auto", "walk", "nodes"])), steps=int(rng.integers(3, 30)),
                lr=float(rng.uniform(0.01, 0.3)), sigma=float(rng.uniform(0.0, 0.3)),
                x0_std=float(rng.choice([0.0, 0.5])), mu_scale=float(rng.uniform(0.5, 3.0)),
                seed=int(rng.integers(0, 2**40)), mu_seed=int(rng.integers(0, 2**40)),
                # drawn from streams of their own, so the other draws of each case are unchanged
                received_sums=bool(np.random.default_rng(5000 + case).integers(0, 2)))
    # regenerated centres take at most 1024 mixture non-zeros (relay_set_objective_generated)
    if c["objective"] == "generated" and np.count_nonzero(c["mix"]) > 1024:
        c["objective"] = "stored"
    return c


@pytest.mark.parametrize("case", range(120))
def test_random_configuration_against_oracle(case):
    c = draw(case)
    n, d, E = c["n"], c["d"], 2 * (c["n"] - 1)
    optimizer = {"sgd": None, "nesterov": ("nesterov", c["beta1"]),
                 "adam": ("adam", c["beta1"], c["beta2"], 1e-2)}[c["opt"]]
    objective = c["objective"]
    run = rs.RelayRun(n, d, c["edges"], device="cuda:0", mode=c["mode"], c0=c["c0"],
                      objective=objective, optimizer=optimizer, algorithm=c["algo"], kernel=c["kernel"],
                      received_sums=c["received_sums"])
    run.init(c["x0_std"], c["seed"], c["mix"], c["mu_scale"], c["mu_seed"], c["sigma"])
    st = oracle.State(n, c["edges"], d, c0=c["c0"])
    st.init(c["x0_std"], c["seed"], c["mix"].astype(np.float64), c["mu_scale"], c["mu_seed"])
    if c["algo"] == "dme":
        run.x.zero_()
        st.x[:] = 0.0
    kw = {}
    if optimizer:
        kw = dict(opt={"nesterov": oracle.OPT_NESTEROV, "adam": oracle.OPT_ADAM}[c["opt"]],
                  beta1=c["beta1"], beta2=c["beta2"] if c["opt"] == "adam" else 0.0,
                  eps=1e-2 if c["opt"] == "adam" else 0.0)
    algo = {"relaysgd": oracle.ALGO_RELAYSGD, "grad": oracle.ALGO_GRAD, "dme": oracle.ALGO_DME}[c["algo"]]
    rng = np.random.default_rng(case)
    lr, sigma = float(np.float32(c["lr"])), float(np.float32(c["sigma"]))
    adam = c["opt"] == "adam"
    bound = np.zeros(d)
    dnoise = generated_input_error(c["mix"], c["mu_scale"], sigma, c["x0_std"])
    for t in range(c["steps"]):
        lost = (rng.random(E) < c["lost_p"]).astype(np.uint8)
        if c["lost_p"] > 0:
            run.set_lost(lost)
        run.step(c["lr"], c["seed"])
        x = st.x.copy()
        st.advance(1, lr, sigma, c["seed"], c["mode"], drop=lost[None, :] if c["lost_p"] > 0 else None,
                   algo=algo, **kw)
        if adam:
            xi = np.stack([oracle.normals(c["seed"], c["c0"], d, row=i, step=t, stream=0) for i in range(n)])
            bound += adam_step_bound(x, st.mu, xi, sigma, st.s1, st.s2, lr, c["beta1"], c["beta2"], 1e-2, t,
                                     dnoise)
    torch.cuda.synchronize()
    info = {k: v for k, v in c.items() if k not in ("edges", "mix")}

    def within(g, r, scale):
        if not adam:
            return parity_error(g, r) <= RTOL
        rms = float(np.sqrt(np.mean(r * r)))
        return bool(np.all(np.abs(g - r) <= RTOL * np.maximum(np.abs(r), rms) + 4.0 * scale * bound[None, :]))

    assert within(run.x[:, :d].double().cpu().numpy(), st.x, 1.0), info
    if E:
        assert within(run.messages[:E, :d].double().cpu().numpy(), st.msg, float(n)), info
        assert np.array_equal(run.counts[:E].cpu().numpy(), st.counts), info
    if c["algo"] == "dme":
        assert np.array_equal(run.trees[0].dme_count.cpu().numpy(), st.dme_count), info
    del run
    gc.collect()
    torch.cuda.empty_cache()
