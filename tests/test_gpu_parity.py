"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle.

Counters bit-exact; models and messages within the parity metric of
tests/gpu_util.py (1e-5).  Small workloads are compared on every coordinate;
the full-size workloads run in full on the GPU, in the launch configuration
bench.py times, and are compared on the first and last coordinates (the
ragged tail included) and on coordinates drawn at random -- every coordinate
of the method evolves independently and the noise is keyed by the absolute
coordinate, so the oracle computes those columns exactly as in a full run.
"""
import gc

import numpy as np
import pytest
import torch

import paper_2110_04175_gb300 as rs
from oracle import oracle
from paper_2110_04175_gb300 import build as rs_build
from paper_2110_04175_gb300 import workloads as wl
from tests import treeutil as tu
from tests.gpu_util import (NORMAL_ABS_ERR, RTOL, c8_sample, compare_ranges, gpu_run, oracle_range, parallel_map,
                             parity_error, record_parity, windows)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    rs_build.build()
    yield
    gc.collect()
    torch.cuda.empty_cache()


def _free():
    gc.collect()
    torch.cuda.empty_cache()


# ------------------------------------------------------------ random streams

def test_initial_model_and_centres_match_oracle_normals():
    d = 4096 + 7
    run = rs.RelayRun(3, d, wl.chain(3), device="cuda:0", objective="stored")
    mix = np.array([[1, 0, 0], [0, 1, 0], [0.25, 0.5, 0.25]], dtype=np.float32)
    run.init(1.0, 1234, mix, 1.5, 99, 0.0)
    torch.cuda.synchronize()
    x = run.x.double().cpu().numpy()
    mu = run.mu.double().cpu().numpy()
    want_x = oracle.fill_x0(3, 1.0, 1234, 0, d)
    want_mu = oracle.fill_mu(3, mix.astype(np.float64), 1.5, 99, 0, d)
    assert parity_error(x[:, :d], want_x) < RTOL
    assert parity_error(mu[:, :d], want_mu) < RTOL
    ragged = slice(d, (d + 3) // 4 * 4)  # the last quad's columns beyond d
    assert np.all(x[:, ragged] == 0) and np.all(mu[:, ragged] == 0)
    edge = (d + 3) // 4 * 4
    assert np.all(run.msg[0][:, :edge].cpu().numpy() == 0)
    assert np.all(run.msg[1][:, :edge].cpu().numpy() == 0)


def test_normal_generator_error_within_derived_bound():
    """The GPU's normals against the oracle's fp64 Box-Muller of the same
    Philox uniforms, on 8.4M draws (the centres of 8 workers over 2^20
    coordinates, mu_i = N_i with an identity mixture): every one within
    gpu_util.NORMAL_ABS_ERR, the bound derived from the GPU's logf,
    sqrt.approx and __sincosf.  The error is small on average too."""
    n, d = 8, 1 << 20
    run = rs.RelayRun(n, d, wl.chain(n), device="cuda:0")
    run.init(0.0, 0, wl.identity_mix(n), 1.0, 12345, 0.0)
    torch.cuda.synchronize()
    g = run.mu[:, :d].double().cpu().numpy()
    want = np.stack(parallel_map(lambda i: oracle.normals(12345, 0, d, row=i, step=0, stream=1), range(n)))
    err = np.abs(g - want)
    assert err.max() <= NORMAL_ABS_ERR, err.max()
    assert err.mean() <= 0.1 * NORMAL_ABS_ERR, err.mean()
    assert np.abs(want).max() > 5.0  # the draws reach the tails, where r is largest


def test_gradient_noise_stream():
    """n = 1, x = mu = 0, lr = 1: one step gives x^1 = -sigma xi^0 exactly as
    the oracle's stream-0 normals, at a non-zero coordinate offset too."""
    for c0, step in ((0, 0), (4096, 7)):
        run = rs.RelayRun(1, 1000, np.zeros((0, 2), np.int32), device="cuda:0", c0=c0)
        run.init(0.0, 77, np.zeros((1, 1), np.float32), 0.0, 0, 0.5)
        run.t = step
        run.step(1.0, 77)
        torch.cuda.synchronize()
        want = -0.5 * oracle.normals(77, c0, 1000, row=0, step=step, stream=0)
        assert parity_error(run.x[0, :1000].double().cpu().numpy(), want) < RTOL


# ------------------------------------------------------------------ counters

@pytest.mark.parametrize("n", [2, 3, 4, 5, 6])
def test_counts_bit_exact_all_small_trees(n):
    trees = list(tu.all_trees(n))
    rng = np.random.default_rng(n)
    if len(trees) > 40:
        trees = [trees[k] for k in rng.choice(len(trees), 40, replace=False)]
    for edges in trees:
        h = rs.relay_create(n, 0, edges)
        E = 2 * (n - 1)
        counts = torch.zeros(E, dtype=torch.int32, device="cuda:0")
        want = np.zeros(E, dtype=np.int32)
        for t in range(tu.diameter(n, edges) + 2):
            rs.relay_step_counts(h, counts)
            oracle.run(n, edges, np.zeros((n, 0)), np.zeros((n, 0)), np.zeros((E, 0)), want, 0, 0,
                       0, t, 1, 0)
            assert np.array_equal(counts.cpu().numpy(), want)


@pytest.mark.parametrize("w", wl.all_workloads(), ids=lambda w: w.name)
def test_counts_bit_exact_workload_trees(w):
    for edges in (w.edges if isinstance(w.edges, list) else [w.edges]):
        h = rs.relay_create(w.n, 0, edges)
        counts = torch.zeros(w.E, dtype=torch.int32, device="cuda:0")
        want = np.zeros(w.E, dtype=np.int32)
        steps = tu.diameter(w.n, edges.tolist()) + 3
        for t in range(steps):
            rs.relay_step_counts(h, counts)
        oracle.run(w.n, edges, np.zeros((w.n, 0)), np.zeros((w.n, 0)), np.zeros((w.E, 0)), want,
                   0, 0, 0, 0, steps, 0)
        assert np.array_equal(counts.cpu().numpy(), want)


# ------------------------------------------------------- full-vector parity

@pytest.mark.parametrize("kernel", ["walk", "nodes"])
@pytest.mark.parametrize("mode", [0, 1])
def test_chain8_d4096_full_100_steps(mode, kernel):
    """The small workload, every coordinate, 100 steps, on each step kernel."""
    w = wl.chain8_d4096()
    run = gpu_run(w, w.steps, mode, kernel=kernel)
    ex, em = compare_ranges(run, w, [(0, w.d)], w.steps, mode, label=f"{w.name}/{kernel}/mode{mode}")
    assert ex <= RTOL and em <= RTOL, (ex, em)


@pytest.mark.parametrize("objective", ["stored", "generated"])
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("shape,n,d", [
    ("single", 1, 4097), ("pair", 2, 33), ("chain", 5, 1), ("chain", 5, 3), ("binary", 7, 5),
    ("star", 9, 131), ("star", 33, 257), ("random", 23, 1031), ("torus", 16, 4099),
    ("star", 256, 67), ("chain", 256, 9),
])
@pytest.mark.parametrize("kernel", ["walk", "nodes"])
def test_small_cases_every_coordinate(shape, n, d, mode, objective, kernel):
    """Edge cases: one worker, one edge, d below one quad, ragged tails, the
    generic high-degree path (stars), the largest supported tree; on each
    step kernel."""
    edges = {"single": np.zeros((0, 2), np.int32), "pair": wl.chain(2), "chain": wl.chain(n),
             "binary": wl.binary_tree(n), "star": wl.star(n), "random": wl.random_tree(n, 4),
             "torus": wl.torus_spanning_tree(4, 4, 2)}[shape]
    w = wl.Workload(f"{shape}{n}", n, edges, d, wl.identity_mix(n), 1.0, 0.1, 0.1, 0.1, 30)
    run = gpu_run(w, w.steps, mode, objective=objective, kernel=kernel)
    ex, em = compare_ranges(run, w, [(0, d)], w.steps, mode)
    assert ex <= RTOL and em <= RTOL, (ex, em)


@pytest.mark.parametrize("kernel", ["walk", "nodes"])
@pytest.mark.parametrize("mix", ["identity", "dirichlet", "dense"])
def test_generated_objective_bit_identical_to_stored(mix, kernel):
    """Regenerating mu in the step kernel (per-row normals or cached centres)
    gives exactly the bits of the stored, pre-filled mu, on both step kernels."""
    n, d = 16, 20_000
    m = {"identity": wl.identity_mix(n), "dirichlet": wl.dirichlet_mix(n, 10, 0.1, seed=3),
         "dense": np.random.default_rng(0).random((n, 24)).astype(np.float32)}[mix]
    w = wl.Workload("mix", n, wl.random_tree(n, 2), d, m, 1.3, 0.05, 0.05, 0.1, 15)
    a = gpu_run(w, w.steps, objective="stored", kernel=kernel)
    b = gpu_run(w, w.steps, objective="generated", kernel=kernel)
    assert torch.equal(a.x, b.x) and torch.equal(a.messages, b.messages)


@pytest.mark.parametrize("n,d", [(16, 9_231), (15, 4_099), (2, 13), (64, 1_001)])
def test_double_binary_trees_match_two_oracle_runs(n, d):
    """Double binary trees (Section 3): tree A owns the first half of the
    coordinates, tree B the rest, both inside one model array.  Each window
    equals an oracle run of its tree on those coordinates, counters included."""
    a, b = wl.double_binary_trees(n)
    w = wl.Workload("dbt", n, a, d, wl.identity_mix(n), 1.0, 0.05, 0.05, 0.1, 25)
    run = rs.RelayRun(n, d, [a, b], device="cuda:0")
    run.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
    for _ in range(w.steps):
        run.step(w.lr, w.seed)
    torch.cuda.synchronize()
    for tr, edges in zip(run.trees, (a, b)):
        wt = wl.Workload("dbt", n, edges, d, w.mix, 1.0, 0.05, 0.05, 0.1, 25)
        st = oracle_range(wt, tr.col0, tr.d, w.steps)
        gx = run.x[:, tr.col0:tr.col0 + tr.d].double().cpu().numpy()
        gm = tr.messages[:tr.E, :tr.d].double().cpu().numpy()
        assert parity_error(gx, st.x) <= RTOL and parity_error(gm, st.msg) <= RTOL
        assert np.array_equal(tr.counts.cpu().numpy(), st.counts)


def test_empty_model_runs_counters_only():
    run = rs.RelayRun(4, 0, wl.chain(4), device="cuda:0")
    run.init(0.0, 0, wl.identity_mix(4), 1.0, 0, 0.1)
    for _ in range(5):
        run.step(0.1, 0)
    torch.cuda.synchronize()
    assert run.counts.cpu().numpy().tolist() == [1, 3, 2, 2, 3, 1]


def test_coordinate_offset_slice_equals_full_run():
    """A handle on coordinates [c0, c0 + len) reproduces those columns of the
    full vector bit for bit (the multi-GPU sharding over d relies on it)."""
    w = wl.Workload("bin15", 15, wl.binary_tree(15), 2000, wl.identity_mix(15), 1.0, 0.1, 0.1,
                    0.1, 20)
    full = gpu_run(w, w.steps)
    part = gpu_run(w, w.steps, d=600, c0=800)
    assert torch.equal(full.x[:, 800:1400], part.x[:, :600])
    assert torch.equal(full.messages[:, 800:1400], part.messages[:, :600])


def test_deterministic_and_resumable():
    """Two runs are bitwise identical; 10 + 10 steps equal 20 steps."""
    w = wl.sweep64("torus")
    w.d = 50_000
    a = gpu_run(w, 20)
    b = gpu_run(w, 10)
    for _ in range(10):
        b.step(w.lr, w.seed)
    torch.cuda.synchronize()
    assert torch.equal(a.x[:, :w.d], b.x[:, :w.d])
    assert torch.equal(a.messages[:, :w.d], b.messages[:, :w.d])
    assert torch.equal(a.counts, b.counts)


def test_streams_are_respected():
    w = wl.chain8_d4096()
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        run = gpu_run(w, 50, stream=s)
    ref = gpu_run(w, 50)
    torch.cuda.synchronize()
    assert torch.equal(run.x, ref.x)


@pytest.mark.parametrize("shape,n,d,kernel,algorithm", [
    ("chain", 8, 4096, "nodes", "relaysgd"), ("binary", 16, 65537, "walk", "relaysgd"),
    ("star", 9, 1031, "walk", "relaysgd"), ("binary", 15, 2053, "nodes", "dme"),
    ("single", 1, 517, "auto", "relaysgd"), ("single", 1, 517, "auto", "dme")])
def test_overlapped_step_launch_equals_separate_launches(shape, n, d, kernel, algorithm):
    """relay_step starts the step kernel as a programmatic dependent of the
    counter kernel; that changes only scheduling, so 60 such steps must equal
    60 steps of relay_step_counts and relay_step_models launched apart, bit
    for bit (including n = 1, where no counter kernel runs unless mean
    estimation needs its counts)."""
    edges = {"chain": wl.chain(n), "binary": wl.binary_tree(n), "star": wl.star(n),
             "single": np.zeros((0, 2), np.int32)}[shape]
    runs = []
    for _ in range(2):
        run = rs.RelayRun(n, d, edges, device="cuda:0", kernel=kernel, algorithm=algorithm)
        run.init(0.1, 5, wl.identity_mix(n), 1.0, 6, 0.1)
        runs.append(run)
    a, b = runs
    for t in range(60):
        a.step(0.05, 5)
        tr = b.trees[0]
        rs.relay_step_counts(tr.h, tr.counts)
        rs.relay_step_models(tr.h, b.x, tr.msg[tr.cur], tr.msg[1 - tr.cur], tr.counts, 0.05, 5, t)
        tr.cur = 1 - tr.cur
    torch.cuda.synchronize()
    assert torch.equal(a.x[:, :d], b.x[:, :d])
    if a.E:
        assert torch.equal(a.messages[:a.E, :d], b.trees[0].messages[:a.E, :d])
        assert torch.equal(a.counts[:a.E], b.trees[0].counts[:a.E])
    if algorithm == "dme":
        assert torch.equal(a.trees[0].dme_count, b.trees[0].dme_count)


# -------------------------------------------------- full-size workloads

FULL = [wl.binary16_resnet20(), wl.chain16_vgg11(), wl.binary32_bert()] + [
    wl.sweep64(s) for s in ("star", "chain", "binary", "torus")]


@pytest.mark.parametrize("w", FULL, ids=lambda w: w.name)
def test_full_size_workload_sampled(w):
    """Full d and the workload's step count on the GPU, in the launch
    configuration bench.py times (stored centres, the automatic kernel
    choice, the workload's rebuild rule).  The oracle checks every coordinate
    of the ResNet-20-sized workload, and on the larger ones the first and
    last 65,536 coordinates plus 1,024 random windows of 1,024."""
    _free()
    run = gpu_run(w, w.steps, objective="stored")
    ranges = windows(w.d) if w.d < 1_000_000 else c8_sample(w.d, seed=w.n)
    ex, em = compare_ranges(run, w, ranges, w.steps, label=w.name)
    del run
    _free()
    assert ex <= RTOL and em <= RTOL, (ex, em)


def test_double16_full_size_sampled():
    """Double binary trees (Section 3) at the VGG-11 size, 200 steps, as
    bench.py runs them (stored centres, both windows in one relay_step_windows
    launch).
    In each tree's coordinate window the oracle runs that tree on the first
    and last 65,536 coordinates and 1,024 random windows of 1,024."""
    _free()
    w = wl.double16_vgg11()
    run = gpu_run(w, w.steps, objective="stored")
    lr, sigma = float(np.float32(w.lr)), float(np.float32(w.sigma))
    for tr, edges in zip(run.trees, w.edges):
        ranges = [(tr.col0 + s, l) for s, l in c8_sample(tr.d, seed=tr.col0 + 1)]

        def oracle_window(r, edges=edges):
            st = oracle.State(w.n, edges, r[1], c0=r[0])
            st.init(w.x0_std, w.seed, w.mix.astype(np.float64), w.mu_scale, w.mu_seed)
            st.advance(w.steps, lr, sigma, w.seed, w.mode)
            return st

        states = parallel_map(oracle_window, ranges)
        gx = np.concatenate([run.x[:, s:s + l].double().cpu().numpy() for s, l in ranges], 1)
        gm = np.concatenate([tr.messages[:tr.E, s - tr.col0:s - tr.col0 + l].double().cpu().numpy()
                             for s, l in ranges], 1)
        ox = np.concatenate([st.x for st in states], 1)
        om = np.concatenate([st.msg for st in states], 1)
        assert np.array_equal(tr.counts[:tr.E].cpu().numpy(), states[0].counts)
        record_parity(f"{w.name}/tree{run.trees.index(tr)}", "x", gx, ox)
        record_parity(f"{w.name}/tree{run.trees.index(tr)}", "messages", gm, om)
        assert parity_error(gx, ox) <= RTOL and parity_error(gm, om) <= RTOL
    del run
    _free()


def test_binary16_resnet20_every_coordinate_mode0():
    """Alg. 1 rebuild on the ResNet-20-sized vector, all 272,474 coordinates,
    oracle on every coordinate for the first 10 steps (the warm-up in which
    nbar < n, where the two rebuild rules differ)."""
    w = wl.binary16_resnet20()
    run = gpu_run(w, 10, mode=0)
    st = oracle_range(w, 0, w.d, 10, 0)
    gx = run.x[:, :w.d].double().cpu().numpy()
    gm = run.messages[:w.E, :w.d].double().cpu().numpy()
    assert parity_error(gx, st.x) <= RTOL
    assert parity_error(gm, st.msg) <= RTOL
    assert np.array_equal(run.counts.cpu().numpy(), st.counts)


def test_double_tree_steps_in_graphs_and_eagerly():
    """Double binary trees: RelayRun.step runs both tree windows in one
    relay_step_windows call, step_forked on forked streams; the eager run,
    a CUDA graph of the same steps replayed once, a forked run and relay_step
    issued window by window on one stream agree bit for bit."""
    n, d = 16, 40_001
    trees = list(wl.double_binary_trees(n))
    runs = []
    for _ in range(4):
        r = rs.RelayRun(n, d, trees, device="cuda:0", kernel="walk")
        r.init(0.1, 3, wl.identity_mix(n), 1.0, 4, 0.1)
        runs.append(r)
    eager, graphed, serial, forked = runs
    for _ in range(25):
        eager.step(0.05, 3)
        forked.step_forked(0.05, 3)
    for _ in range(5):
        graphed.step(0.05, 3)
    g = graphed.capture(20, 0.05, 3)
    g.replay()
    for t in range(25):
        for tr in serial.trees:
            rs.relay_step(tr.h, serial._x(tr), tr.msg[tr.cur], tr.msg[1 - tr.cur], tr.counts, 0.05, 3, t)
            tr.cur = 1 - tr.cur
    torch.cuda.synchronize()
    for other in (graphed, serial, forked):
        assert torch.equal(other.x[:, :d], eager.x[:, :d])
        for ta, tb in zip(other.trees, eager.trees):
            assert torch.equal(ta.messages[:ta.E, :ta.d], tb.messages[:tb.E, :tb.d])
            assert torch.equal(ta.counts, tb.counts)


def test_captured_graph_equals_eager_steps():
    """A CUDA graph of K captured steps, replayed once, gives the eager run."""
    w = wl.chain8_d4096()
    eager = gpu_run(w, 30)
    run = rs.RelayRun(w.n, w.d, w.edges, device="cuda:0")
    run.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
    for _ in range(10):
        run.step(w.lr, w.seed)
    g = run.capture(20, w.lr, w.seed)
    g.replay()
    torch.cuda.synchronize()
    assert run.t == 30
    assert torch.equal(run.x[:, :w.d], eager.x[:, :w.d])
    assert torch.equal(run.messages[:, :w.d], eager.messages[:, :w.d])
    assert torch.equal(run.counts, eager.counts)


@pytest.mark.parametrize("optimizer,algorithm", [(None, "relaysgd"), (("adam", 0.9, 0.99, 1e-8), "relaysgd"),
                                                 (None, "dme")])
def test_checkpoint_resume_is_bit_exact(optimizer, algorithm):
    """Save the full state after k steps, restore it into a fresh run, take k
    more steps: identical to 2k uninterrupted steps."""
    w = wl.sweep64("star")
    w.d = 20_000
    kw = dict(device="cuda:0", optimizer=optimizer, algorithm=algorithm)
    a = rs.RelayRun(w.n, w.d, w.edges, **kw)
    a.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
    for _ in range(12):
        a.step(w.lr, w.seed)
    b = rs.RelayRun(w.n, w.d, w.edges, **kw)
    b.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
    for _ in range(6):
        b.step(w.lr, w.seed)
    sd = b.state_dict()
    c = rs.RelayRun(w.n, w.d, w.edges, **kw)
    c.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
    c.load_state_dict(sd)
    for _ in range(6):
        c.step(w.lr, w.seed)
    torch.cuda.synchronize()
    assert torch.equal(a.x[:, :w.d], c.x[:, :w.d])
    assert torch.equal(a.messages[:, :w.d], c.messages[:, :w.d])
    assert torch.equal(a.counts, c.counts)
    if algorithm == "dme":
        assert torch.equal(a.trees[0].dme_count, c.trees[0].dme_count)
