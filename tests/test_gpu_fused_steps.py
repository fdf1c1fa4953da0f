"""relay_steps (k steps in one launch, the state kept on chip between them)
against k relay_step calls, and against the oracle.

Equivalence: two identical runs, one advanced by relay_step calls and one by
relay_steps, must hold the same models, both message buffers, counters,
mean-estimation counts and optimiser state bit for bit after every chunk.
The chunks (1, 2, 3, 64, 65, 130 steps) cover a single step, the odd and even
buffer parities, one full launch of 64 steps and runs split over two and three
launches.  The configurations cover every degree path (chains, binary trees,
a star's wide hub, random trees up to 200 workers), both rebuild rules, the
three local optimisers, the three algorithms, lost messages, a coordinate
offset, ragged vector lengths, one worker, and the double binary trees.
Parity: relay_steps alone against the fp64 oracle (1e-5, counters exact).
"""
import gc

import numpy as np
import pytest
import torch

import paper_2110_04175_gb300 as rs
from oracle import oracle
from paper_2110_04175_gb300 import build as rs_build
from paper_2110_04175_gb300 import workloads as wl
from tests.gpu_util import RTOL, parity_error

pytestmark = pytest.mark.gpu

CHUNKS = [1, 2, 3, 64, 65, 130]


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    rs_build.build()
    yield
    gc.collect()
    torch.cuda.empty_cache()


CASES = {
    "chain8_d4096": dict(n=8, edges=wl.chain(8), d=4096),
    "binary16_ragged_offset_alg1": dict(n=16, edges=wl.binary_tree(16), d=4097, c0=4000, mode=0),
    "star20_lost": dict(n=20, edges=wl.star(20), d=3001, lost_p=0.2),
    # received sums off: under "nodes" the multi-step kernel's wide-node path
    "star20_lost_plain": dict(n=20, edges=wl.star(20), d=3001, lost_p=0.2, received_sums=False),
    "star64_dme_lost_plain": dict(n=64, edges=wl.star(64), d=513, algorithm="dme", lost_p=0.1,
                                  received_sums=False),
    "random100_nesterov_generated": dict(n=100, edges=wl.random_tree(100, 7), d=333,
                                         optimizer=("nesterov", 0.9), objective="generated"),
    "binary200_adam": dict(n=200, edges=wl.binary_tree(200), d=65, optimizer=("adam", 0.9, 0.999, 1e-8)),
    "torus64_grad": dict(n=64, edges=wl.torus_spanning_tree(8, 8), d=1000, algorithm="grad"),
    "star64_dme_lost": dict(n=64, edges=wl.star(64), d=513, algorithm="dme", lost_p=0.1),
    "one_worker_dme": dict(n=1, edges=wl.chain(1), d=100, algorithm="dme"),
    "one_worker_adam": dict(n=1, edges=wl.chain(1), d=37, optimizer=("adam", 0.8, 0.99, 1e-3)),
    "pair_nesterov_alg1": dict(n=2, edges=wl.chain(2), d=9, mode=0, optimizer=("nesterov", 0.5)),
    "chain5_generated_lost": dict(n=5, edges=wl.chain(5), d=2001, objective="generated", lost_p=0.3),
    "double16_trees": dict(n=16, edges=list(wl.double_binary_trees(16)), d=9001),
}


def make_run(c, seed=3, kernel="auto"):
    run = rs.RelayRun(c["n"], c["d"], c["edges"], device="cuda:0", mode=c.get("mode", 1), c0=c.get("c0", 0),
                      objective=c.get("objective", "stored"), optimizer=c.get("optimizer"),
                      algorithm=c.get("algorithm", "relaysgd"), kernel=kernel,
                      received_sums=c.get("received_sums", True))
    n = c["n"]
    mix = wl.dirichlet_mix(n, 5, 0.3, seed) if n > 2 else wl.identity_mix(n)
    run.init(0.5, seed, mix, 1.5, seed + 1, 0.2)
    if c.get("algorithm") == "dme":
        run.x.zero_()
    if c.get("lost_p"):
        rng = np.random.default_rng(seed)
        for t, tr in enumerate(run.trees):
            run.set_lost((rng.random(tr.E) < c["lost_p"]).astype(np.uint8), tree=t)
    return run


def state_of(run):
    out = {"x": run.x[:, :run.d].clone()}
    for k, st in enumerate(run.state):
        out[f"s{k + 1}"] = st[:, :run.d].clone()
    for t, tr in enumerate(run.trees):
        out[f"t{t}.cur"] = tr.cur
        if tr.E:
            rows = rs.relay_message_rows(tr.h)  # the messages and any received-sum rows
            for b in (0, 1):
                out[f"t{t}.msg{b}"] = tr.msg[b][:rows, :tr.d].clone()
            out[f"t{t}.counts"] = tr.counts[:tr.E].clone()
        if tr.dme_count is not None:
            out[f"t{t}.dme"] = tr.dme_count.clone()
    return out


@pytest.mark.parametrize("kernel", ["auto", "nodes"])
@pytest.mark.parametrize("name", sorted(CASES))
def test_steps_equal_step_calls_bit_for_bit(name, kernel):
    """kernel="nodes" forces the multi-step kernel for relay_steps (the wide-node
    path included, with received sums off) and the node kernel for relay_step;
    under "auto", and with received sums on, the stars take the per-step
    fallback."""
    c = CASES[name]
    a, b = make_run(c, kernel=kernel), make_run(c, kernel=kernel)
    lr, seed = 0.05, 11
    for k in CHUNKS:
        for _ in range(k):
            a.step(lr, seed)
        b.steps(k, lr, seed)
        torch.cuda.synchronize()
        sa, sb = state_of(a), state_of(b)
        assert sa.keys() == sb.keys()
        for key in sa:
            if isinstance(sa[key], int):
                assert sa[key] == sb[key], (name, k, key)
            else:
                assert torch.equal(sa[key], sb[key]), (name, k, key)
        assert a.t == b.t


def test_steps_started_at_a_later_step_and_mixed_with_step_calls():
    """relay_steps continues a run wherever relay_step left it (t0 > 0, either
    buffer parity), and relay_step continues after it."""
    c = CASES["binary16_ragged_offset_alg1"]
    a, b = make_run(c, seed=5), make_run(c, seed=5)
    for plan in ([("step", 3), ("steps", 5), ("step", 1), ("steps", 70), ("step", 2)]):
        kind, k = plan
        for _ in range(k):
            a.step(0.1, 2)
        if kind == "step":
            for _ in range(k):
                b.step(0.1, 2)
        else:
            b.steps(k, 0.1, 2)
    torch.cuda.synchronize()
    sa, sb = state_of(a), state_of(b)
    for key in sa:
        if not isinstance(sa[key], int):
            assert torch.equal(sa[key], sb[key]), key


def test_steps_inside_a_cuda_graph():
    c = CASES["chain8_d4096"]
    a, b = make_run(c), make_run(c)
    for _ in range(100):
        a.step(0.1, 4)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        b.steps(100, 0.1, 4, side)
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(a.x[:, :c["d"]], b.x[:, :c["d"]])
    assert torch.equal(a.messages[:a.E, :c["d"]], b.messages[:b.E, :c["d"]])


@pytest.mark.parametrize("shape,n,d,mode", [("chain", 8, 4096, 1), ("binary", 16, 4097, 0), ("star", 12, 1001, 1)])
def test_steps_against_oracle(shape, n, d, mode):
    edges = {"chain": wl.chain, "binary": wl.binary_tree, "star": wl.star}[shape](n)
    steps, lr, sigma, seed, mu_seed = 100, 0.1, 0.1, 7, 8
    mix = wl.identity_mix(n)
    run = rs.RelayRun(n, d, edges, device="cuda:0", mode=mode)
    run.init(0.5, seed, mix, 2.0, mu_seed, sigma)
    run.steps(steps, lr, seed)
    torch.cuda.synchronize()
    st = oracle.State(n, edges, d)
    st.init(0.5, seed, mix.astype(np.float64), 2.0, mu_seed)
    st.advance(steps, float(np.float32(lr)), float(np.float32(sigma)), seed, mode)
    assert parity_error(run.x[:, :d].double().cpu().numpy(), st.x) <= RTOL
    assert parity_error(run.messages[:run.E, :d].double().cpu().numpy(), st.msg) <= RTOL
    assert np.array_equal(run.counts[:run.E].cpu().numpy(), st.counts)


@pytest.mark.parametrize("name", ["chain16_d9231114_dirichlet", "binary32_d110000000"])
def test_full_size_steps_equal_step_calls(name):
    """At the sizes bench.py times, every CTA of the multi-step kernel carries
    hundreds of quad blocks in turn (its loop refills the message buffer and
    reuses the rebuild factors), which the small cases above never reach:
    70 steps (two launches) through relay_steps equal 70 relay_step calls bit
    for bit there too -- models, both message buffers and counters."""
    w = wl.by_name(name)
    runs = []
    for _ in range(2):
        run = rs.RelayRun(w.n, w.d, w.edges, device="cuda:0", mode=w.mode)
        run.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
        runs.append(run)
    a, b = runs
    assert rs.relay_get_steps_kernel(b.h) == rs.RELAY_KERNEL_FUSED
    for _ in range(70):
        a.step(w.lr, w.seed)
    b.steps(70, w.lr, w.seed)
    torch.cuda.synchronize()
    assert torch.equal(a.x[:, :w.d], b.x[:, :w.d])
    for k in (0, 1):
        assert torch.equal(a.msg[k][:a.E, :w.d], b.msg[k][:b.E, :w.d]), k
    assert torch.equal(a.counts[:a.E], b.counts[:b.E])
    assert a.cur == b.cur
    del a, b, runs
    gc.collect()
    torch.cuda.empty_cache()
