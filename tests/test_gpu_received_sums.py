"""Received sums (relay_set_received_sums) on the GPU.

A wide node i (degree > 4) sends neighbour j the message x_i^{t+1/2} +
S_i^{t-1} - m^{t-1}_{j->i}, with S_i^{t-1} the sum of the messages it received
at step t-1 (Alg. 1's rebuild sum).  With received sums on, each message buffer
carries S_i after its E message rows, so every incoming row is read once.

Checked here:
- each sum row equals the fp32 sum of the wide node's received messages, added
  from zero in the program's rebuild order, bit for bit, on both step kernels
  and after every step;
- the models and messages match the fp64 oracle on every coordinate (1e-5)
  with received sums on, as they do with them off, on stars up to 256 workers
  and trees with several adjacent wide nodes, under both rebuild rules, every
  algorithm, local Nesterov and lost messages;
- the counters are those of the plain path.
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


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    rs_build.build()
    yield
    gc.collect()
    torch.cuda.empty_cache()


def _twin():
    """Two adjacent hubs with leaves: a wide node whose DFS parent is wide."""
    return np.array([(0, 1)] + [(0, k) for k in range(2, 8)] + [(1, k) for k in range(8, 14)], np.int32)


def _chain3():
    """Three hubs along a path, with narrow nodes and a short branch between."""
    e = ([(0, 1), (1, 2), (2, 3), (3, 4)] + [(0, k) for k in range(5, 10)] + [(2, k) for k in range(10, 15)] +
         [(4, k) for k in range(15, 21)] + [(15, 21), (21, 22)])
    return np.array(e, np.int32)


TREES = {
    "star9": lambda: wl.star(9),
    "star33_hub5": lambda: wl.star(33, hub=5),
    "star256": lambda: wl.star(256),
    "twin": _twin,
    "chain3": _chain3,
}


def _n(edges) -> int:
    return int(np.asarray(edges).max()) + 1


def _host_sums(run, tr):
    """Per wide node, its sum row recomputed on the host in float32: zero plus
    its received messages in the program's rebuild order."""
    _, _, node, pos = rs.relay_program(tr.h)
    msg = tr.messages.cpu().numpy()
    E = tr.E
    out = {}
    for i in range(run.n):
        row = int(node[i][11])
        if row < 0:
            continue
        s = np.zeros(msg.shape[1], np.float32)
        for k in range(int(node[i][0])):
            s = s + msg[int(pos[int(node[i][1]) + k][3])]
        out[E + row] = s
    return out


@pytest.mark.parametrize("kernel", ["walk", "nodes"])
@pytest.mark.parametrize("tree", ["star9", "star256", "twin", "chain3"])
def test_sum_rows_are_the_received_sums_bit_for_bit(tree, kernel):
    edges = TREES[tree]()
    n, d = _n(edges), 1031
    run = rs.RelayRun(n, d, edges, device="cuda:0", kernel=kernel)
    rng = np.random.default_rng(5)
    run.init(0.3, 7, wl.identity_mix(n), 1.0, 8, 0.1)
    tr = run.trees[0]
    assert rs.relay_message_rows(tr.h) > tr.E
    for t in range(6):
        run.set_lost((rng.random(tr.E) < 0.15).astype(np.uint8))
        run.step(0.1, 7)
        torch.cuda.synchronize()
        got = tr.messages.cpu().numpy()
        for row, want in _host_sums(run, tr).items():
            assert np.array_equal(got[row, :d], want[:d]), (tree, kernel, t, row)


CASES = [
    # tree, d, mode, algorithm, optimizer, lost probability
    ("star9", 131, 1, "relaysgd", None, 0.0),
    ("star9", 4099, 0, "relaysgd", None, 0.0),
    ("star33_hub5", 257, 1, "relaysgd", ("nesterov", 0.9), 0.0),
    ("star256", 67, 1, "relaysgd", None, 0.0),
    ("star256", 67, 0, "relaysgd", None, 0.1),
    ("twin", 1031, 1, "relaysgd", None, 0.2),
    ("twin", 1031, 0, "grad", None, 0.0),
    ("chain3", 2053, 1, "dme", None, 0.1),
    ("chain3", 2053, 1, "relaysgd", None, 0.0),
]


@pytest.mark.parametrize("kernel", ["walk", "nodes"])
@pytest.mark.parametrize("tree,d,mode,algorithm,optimizer,lost_p", CASES)
def test_received_sums_against_oracle_every_coordinate(tree, d, mode, algorithm, optimizer, lost_p, kernel):
    """With and without received sums, the models, messages and counters match
    the oracle; the counters of the two paths are identical."""
    edges = TREES[tree]()
    n, steps, lr, sigma, seed = _n(edges), 30, 0.05, 0.1, 9
    mix = wl.dirichlet_mix(n, 4, 0.5, 3)
    lost_rng = np.random.default_rng(11)
    E = 2 * (n - 1)
    lost = (lost_rng.random((steps, E)) < lost_p).astype(np.uint8)
    results = []
    for sums in (True, False):
        run = rs.RelayRun(n, d, edges, device="cuda:0", mode=mode, algorithm=algorithm, optimizer=optimizer,
                          kernel=kernel, received_sums=sums)
        run.init(0.2, seed, mix, 1.2, seed + 1, sigma)
        if algorithm == "dme":
            run.x.zero_()
        for t in range(steps):
            run.set_lost(lost[t] if lost_p > 0 else None)
            run.step(lr, seed)
        torch.cuda.synchronize()
        results.append((run.x[:, :d].double().cpu().numpy(), run.messages[:E, :d].double().cpu().numpy(),
                        run.counts[:E].cpu().numpy(),
                        None if run.trees[0].dme_count is None else run.trees[0].dme_count.cpu().numpy()))
        del run
    st = oracle.State(n, edges, d)
    st.init(0.2, seed, mix.astype(np.float64), 1.2, seed + 1)
    algo = {"relaysgd": oracle.ALGO_RELAYSGD, "grad": oracle.ALGO_GRAD, "dme": oracle.ALGO_DME}[algorithm]
    if algo == oracle.ALGO_DME:
        st.x[:] = 0.0  # running sums start at zero
    kw = dict(opt=oracle.OPT_NESTEROV, beta1=optimizer[1]) if optimizer else {}
    st.advance(steps, float(np.float32(lr)), float(np.float32(sigma)), seed, mode,
               drop=lost if lost_p > 0 else None, algo=algo, **kw)
    for x, m, c, dme in results:
        assert parity_error(x, st.x) <= RTOL
        assert parity_error(m, st.msg) <= RTOL
        assert np.array_equal(c, st.counts)
        if dme is not None:
            assert np.array_equal(dme, st.dme_count)
    assert np.array_equal(results[0][2], results[1][2])
