"""The node-parallel step kernel (RELAY_KERNEL_NODES: one thread per worker
and quad, messages exchanged through shared memory) against the walk kernel
(RELAY_KERNEL_WALK) bit for bit over every feature, and against the oracle.

Both kernels form each message and each rebuild sum in the same order, so
every model, message, counter and optimiser-state value must be identical;
the oracle comparisons hold the node kernel to the same parity bar as the
walk kernel on its own.
"""
import gc

import numpy as np
import pytest
import torch

import paper_2110_04175_gb300 as rs
from oracle import oracle
from paper_2110_04175_gb300 import build as rs_build
from paper_2110_04175_gb300 import workloads as wl
from tests.gpu_util import RTOL, compare_ranges, parity_error, windows

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    rs_build.build()
    yield
    gc.collect()
    torch.cuda.empty_cache()


SHAPES = {
    "single": (1, lambda: np.zeros((0, 2), np.int32)),
    "pair": (2, lambda: wl.chain(2)),
    "chain8": (8, lambda: wl.chain(8)),
    "star9": (9, lambda: wl.star(9)),            # hub of degree 8: the wide path
    "binary15": (15, lambda: wl.binary_tree(15)),
    "random20": (20, lambda: wl.random_tree(20, 3)),
    "torus16": (16, lambda: wl.torus_spanning_tree(4, 4, 0)),
    "star64": (64, lambda: wl.star(64)),
    "random100": (100, lambda: wl.random_tree(100, 5)),  # one quad per CTA
    "chain256": (256, lambda: wl.chain(256)),            # 256 threads per CTA
}

OPTIMIZERS = {None: None, "nesterov": ("nesterov", 0.9), "adam": ("adam", 0.9, 0.99, 1e-8)}


def _run(kernel, n, edges, d, steps=12, mode=1, objective="stored", optimizer=None,
         algorithm="relaysgd", lost_p=0.0, mix=None, seed=4, received_sums=True):
    run = rs.RelayRun(n, d, edges, device="cuda:0", mode=mode, objective=objective,
                      optimizer=OPTIMIZERS[optimizer], algorithm=algorithm, kernel=kernel,
                      received_sums=received_sums)
    mix = wl.identity_mix(n) if mix is None else mix
    run.init(0.1, seed, mix, 1.0, seed + 1, 0.1)
    if algorithm == "dme":
        run.x.zero_()
    rng = np.random.default_rng(seed)
    for _ in range(steps):
        if lost_p > 0:
            for k, tr in enumerate(run.trees):
                run.set_lost((rng.random(tr.E) < lost_p).astype(np.uint8), tree=k)
        run.step(0.05, seed)
    torch.cuda.synchronize()
    return run


def _assert_identical(a, b, d):
    assert torch.equal(a.x[:, :d], b.x[:, :d])
    for sa, sb in zip(a.state, b.state):
        assert torch.equal(sa[:, :d], sb[:, :d])
    for ta, tb in zip(a.trees, b.trees):
        rows = rs.relay_message_rows(ta.h)  # the messages and any received-sum rows
        assert torch.equal(ta.messages[:rows, :ta.d], tb.messages[:rows, :tb.d])
        assert torch.equal(ta.counts[:ta.E], tb.counts[:tb.E])
        if ta.dme_count is not None:
            assert torch.equal(ta.dme_count, tb.dme_count)


def _both(n, edges, d, **kw):
    a = _run("walk", n, edges, d, **kw)
    b = _run("nodes", n, edges, d, **kw)
    _assert_identical(a, b, d)
    del a, b
    gc.collect()
    torch.cuda.empty_cache()


@pytest.mark.parametrize("objective", ["stored", "generated"])
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("shape", list(SHAPES))
def test_nodes_equal_walk_every_shape(shape, mode, objective):
    n, edges = SHAPES[shape]
    for d in (1, 13, 4099):
        _both(n, edges(), d, mode=mode, objective=objective)


@pytest.mark.parametrize("shape", ["chain8", "star9", "binary15", "star64"])
@pytest.mark.parametrize("optimizer,algorithm,lost_p", [
    ("nesterov", "relaysgd", 0.0), ("adam", "relaysgd", 0.0), (None, "grad", 0.0),
    (None, "dme", 0.0), (None, "relaysgd", 0.2), ("adam", "relaysgd", 0.2), (None, "dme", 0.2)])
def test_nodes_equal_walk_every_feature(shape, optimizer, algorithm, lost_p):
    n, edges = SHAPES[shape]
    _both(n, edges(), 2053, mode=0 if lost_p == 0 else 1, optimizer=optimizer,
          algorithm=algorithm, lost_p=lost_p)


@pytest.mark.parametrize("objective", ["stored", "generated"])
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("shape", ["star9", "star64"])
def test_nodes_equal_walk_wide_nodes_without_received_sums(shape, mode, objective):
    """The wide path that reads every incoming row (received sums off)."""
    n, edges = SHAPES[shape]
    for d in (13, 4099):
        _both(n, edges(), d, mode=mode, objective=objective, received_sums=False)
    _both(n, edges(), 2053, optimizer="adam", lost_p=0.2, received_sums=False)
    _both(n, edges(), 2053, algorithm="dme", lost_p=0.2, received_sums=False)


@pytest.mark.parametrize("mix", ["dirichlet", "dense"])
def test_nodes_equal_walk_regenerated_mixtures(mix):
    """The walk caches the K regenerated centres per quad; the node kernel
    forms them per row: the same normals mixed in the same order."""
    n = 12
    m = (wl.dirichlet_mix(n, 10, 0.1, 3) if mix == "dirichlet"
         else np.random.default_rng(2).random((n, 6)).astype(np.float32))
    _both(n, wl.binary_tree(n), 3001, objective="generated", mix=m)


def test_nodes_equal_walk_double_binary_trees():
    a, b = wl.double_binary_trees(16)
    _both(16, [a, b], 9231, lost_p=0.1)


@pytest.mark.parametrize("shape", ["binary15", "star64"])
def test_nodes_equal_walk_many_blocks(shape):
    """Enough quads that every CTA loops over several blocks."""
    n, edges = SHAPES[shape]
    _both(n, edges(), 1_000_003, steps=4)


@pytest.mark.parametrize("mode", [0, 1])
def test_nodes_chain8_d4096_full_100_steps_against_oracle(mode):
    """The 8-worker chain at d = 4096, every coordinate, 100 steps."""
    w = wl.chain8_d4096()
    run = rs.RelayRun(w.n, w.d, w.edges, device="cuda:0", mode=mode, kernel="nodes")
    run.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
    for _ in range(w.steps):
        run.step(w.lr, w.seed)
    torch.cuda.synchronize()
    st = oracle.State(w.n, w.edges, w.d)
    st.init(w.x0_std, w.seed, w.mix.astype(np.float64), w.mu_scale, w.mu_seed)
    st.advance(w.steps, float(np.float32(w.lr)), float(np.float32(w.sigma)), w.seed, mode)
    assert parity_error(run.x[:, :w.d].double().cpu().numpy(), st.x) <= RTOL
    assert parity_error(run.messages[:run.E, :w.d].double().cpu().numpy(), st.msg) <= RTOL
    assert np.array_equal(run.counts[:run.E].cpu().numpy(), st.counts)


def test_nodes_binary16_resnet20_every_coordinate_against_oracle():
    """The 16-worker binary tree at d = 272,474 (ResNet-20-sized), 500 steps,
    on the node kernel with regenerated centres (the full-size parity test
    covers the stored ones), every coordinate checked by the oracle."""
    w = wl.binary16_resnet20()
    run = rs.RelayRun(w.n, w.d, w.edges, device="cuda:0", mode=w.mode, kernel="nodes",
                      objective="generated")
    run.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
    for _ in range(w.steps):
        run.step(w.lr, w.seed)
    torch.cuda.synchronize()
    ex, em = compare_ranges(run, w, windows(w.d), w.steps)
    assert ex <= RTOL and em <= RTOL, (ex, em)
