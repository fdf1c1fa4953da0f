"""CPU checks of the library's host logic (no GPU needed).

The fused kernel follows a visit program built on the host (tree walk,
shared-memory slot assignment).  Here the program is read back through the
C ABI and executed in float64 with the kernel's exact sequence of slot reads
and writes -- every write must land in a free slot, every read in a live
one -- and the result is compared with the oracle.  A wrong slot assignment,
parent link or finalisation point fails here before any GPU time is spent.
"""
import ctypes
import re

import numpy as np
import pytest

import paper_2110_04175_gb300 as rs
from oracle import oracle
from paper_2110_04175_gb300 import build as rs_build
from paper_2110_04175_gb300 import workloads as wl
from tests import treeutil as tu


@pytest.fixture(scope="module", autouse=True)
def _built():
    rs_build.build()


REG_DEG = 4


def run_program(h, n, x, mu, msg_in, counts_old, lr, sigma, seed, step, mode, c0=0, lost=None):
    """One step executed the way relay_counts_kernel + relay_models_kernel do
    (lost: E flags of messages lost in transit, or None).  With received sums
    on (a wide node's rsum_row >= 0), msg_in and the result carry the sum
    rows after the E message rows."""
    lost = np.zeros(2 * (n - 1), dtype=bool) if lost is None else np.asarray(lost, dtype=bool)
    nslots, order, node, pos = rs.relay_program(h)
    E = 2 * (n - 1)
    sums = bool(n > 0 and (node[:, 11] >= 0).any())
    rows = rs.relay_message_rows(h)
    assert rows == E + int((node[:, 11] >= 0).sum())
    src, dst = rs.relay_edges(h)
    # counters
    counts = np.zeros(E, dtype=np.int32)
    for e in range(E):
        deg, pb = node[src[e]][0], node[src[e]][1]
        counts[e] = 0 if lost[e] else 1 + sum(counts_old[pos[pb + s][0]] for s in range(deg)
                                              if pos[pb + s][0] != (e ^ 1))
    nbar = [1 + sum(counts[pos[node[i][1] + s][0]] for s in range(node[i][0])) for i in range(n)]
    if mode == 0:
        scale = [1.0 / nb for nb in nbar]
        fill = [0.0] * n
    else:
        scale = [1.0 / n] * n
        fill = [float(n - nb) for nb in nbar]
    L = x.shape[1]
    slots = [None] * nslots
    msg_out = np.full((rows, L), np.nan)
    xnew = np.full((n, L), np.nan)
    visited = set()

    def write(s, v):
        assert 0 <= s < nslots and slots[s] is None, f"slot {s} clobbered"
        slots[s] = v

    def take(s):
        assert slots[s] is not None, f"slot {s} read while free"
        v = slots[s]
        slots[s] = None
        return v

    def to_parent(rec, out):
        par, pacc, finp = rec[7], rec[5], rec[6]
        assert par in visited
        acc = take(pacc) + out
        if sums and rec[9] & 1:            # the wide parent's received sum S_p^t
            rsum = take(node[par][10]) + out
            if finp >= 0:
                msg_out[E + node[par][11]] = rsum
            else:
                write(node[par][10], rsum)
        if finp >= 0:
            assert finp == par
            xnew[finp] = acc * scale[finp]
            if node[par][8] >= 0:          # the wide parent's total dies with it
                take(node[par][8])
        else:
            write(pacc, acc)

    for i in order:
        visited.add(i)
        rec = node[i]
        deg, pb, ppos, recv, accs, tot, flags = rec[0], rec[1], rec[2], rec[3], rec[4], rec[8], rec[9]
        z = oracle.normals(seed, c0, L, i, step, 0)
        xh = x[i] - lr * ((x[i] - mu[i]) + sigma * z)
        acc = xh.copy()
        if mode == 1:
            acc = fill[i] * x[i] + xh
        m_par = np.zeros(L)
        if recv >= 0:
            if flags & 1:
                # the parent is wide: recv holds its total, which stays live
                assert slots[recv] is not None
                m = slots[recv] - msg_in[pos[pb + ppos][1]]
                m = 0 * m if lost[pos[pb + ppos][0]] else m
                msg_out[pos[pb + ppos][0]] = m
                m_par = m
            else:
                m_par = take(recv)
            acc = acc + m_par
        if sums and deg > REG_DEG:
            write(rec[10], 0 + m_par)      # S_i^t starts with the DFS parent's message
        if 0 < deg <= REG_DEG:
            m = [msg_in[pos[pb + s][0]] for s in range(deg)]
            for s in range(deg):
                out = xh + sum((m[r] for r in range(deg) if r != s), np.zeros(L))
                out = 0 * out if lost[pos[pb + s][1]] else out
                msg_out[pos[pb + s][1]] = out
                if s == ppos:
                    to_parent(rec, out)
                else:
                    write(pos[pb + s][2], out)
        elif deg > REG_DEG:
            if sums:                       # T_i = x^{t+1/2} + S_i^{t-1}, one row
                total = xh + msg_in[E + rec[11]]
            else:
                total = xh + sum(msg_in[pos[pb + s][0]] for s in range(deg))
            if ppos >= 0:
                out = total - msg_in[pos[pb + ppos][0]]
                out = 0 * out if lost[pos[pb + ppos][1]] else out
                msg_out[pos[pb + ppos][1]] = out
                to_parent(rec, out)
            write(tot, total)
        if accs < 0:
            xnew[i] = acc * scale[i]
        else:
            write(accs, acc)
    assert all(s is None for s in slots), "slots left live after the walk"
    assert not np.isnan(xnew).any() and not np.isnan(msg_out).any()
    return xnew, msg_out, counts, nslots


def check_tree(n, edges, mode, steps=3, L=3, seed=1, p_lost=0.0, sums=False):
    h = rs.relay_create(n, L, edges)
    rs.relay_set_received_sums(h, sums)
    lost_rng = np.random.default_rng(1000 + n)
    rng = np.random.default_rng(n)
    mu = rng.normal(size=(n, L))
    x = np.tile(rng.normal(size=L), (n, 1))
    E = 2 * (n - 1)
    st = oracle.State(n, edges, L)
    st.x = x.copy()
    st.mu = mu.copy()
    msg = np.zeros((rs.relay_message_rows(h), L))
    counts = np.zeros(E, dtype=np.int32)
    src, dst = rs.relay_edges(h)
    _, _, node, _ = rs.relay_program(h)
    for t in range(steps):
        lost = (lost_rng.random(E) < p_lost).astype(np.uint8)
        x, msg, counts, nslots = run_program(h, n, x, mu, msg, counts, 0.3, 0.2, seed, t, mode,
                                             lost=lost)
        st.advance(1, 0.3, 0.2, seed, mode, drop=lost[None, :] if p_lost > 0 else None)
        assert np.array_equal(counts, st.counts)
        assert np.allclose(x, st.x, rtol=1e-12, atol=1e-12)
        assert np.allclose(msg[:E], st.msg, rtol=1e-12, atol=1e-12)
        for i in range(n):  # a sum row holds the sum of the wide node's received messages
            if node[i][11] >= 0:
                assert np.allclose(msg[E + node[i][11]], msg[:E][dst == i].sum(axis=0), rtol=1e-12, atol=1e-12)
    return nslots


@pytest.mark.parametrize("sums", [False, True])
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("n", [1, 2, 3, 4, 5, 6])
def test_program_matches_oracle_small_trees(n, mode, sums):
    trees = list(tu.all_trees(n))
    rng = np.random.default_rng(n)
    if len(trees) > 80:
        trees = [trees[k] for k in rng.choice(len(trees), 80, replace=False)]
    for edges in trees:
        check_tree(n, edges, mode, sums=sums)


def _wide_trees():
    """Trees with several wide nodes next to each other and next to narrow ones."""
    # two hubs joined by an edge, each with leaves; a hub whose parent is a hub
    twin = [(0, 1)] + [(0, k) for k in range(2, 8)] + [(1, k) for k in range(8, 14)]
    # a chain of three hubs with a narrow node and a subtree between
    chain3 = ([(0, 1), (1, 2), (2, 3), (3, 4)] + [(0, k) for k in range(5, 10)] +
              [(2, k) for k in range(10, 15)] + [(4, k) for k in range(15, 21)] + [(15, 21), (21, 22)])
    return {"twin": np.array(twin, np.int32), "chain3": np.array(chain3, np.int32)}


@pytest.mark.parametrize("sums", [False, True])
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("shape", ["star", "chain", "binary", "torus", "random40", "star9", "twin", "chain3"])
def test_program_matches_oracle_workload_trees(shape, mode, sums):
    trees = {"star": wl.star(64), "chain": wl.chain(64), "binary": wl.binary_tree(64),
             "torus": wl.torus_spanning_tree(8, 8, 0), "random40": wl.random_tree(40, 9),
             "star9": wl.star(9, hub=4), **_wide_trees()}
    edges = trees[shape]
    n = int(edges.max()) + 1
    check_tree(n, edges, mode, steps=2 if n > 30 else 5, L=2, sums=sums)


@pytest.mark.parametrize("sums", [False, True])
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("shape", ["star", "binary", "random40", "star9", "chain", "twin", "chain3"])
def test_program_with_lost_messages_matches_oracle(shape, mode, sums):
    """Lost messages (Section 4.4) are zeroed where the kernel zeroes them --
    including the messages a wide node's children form from its total, and
    the received sums add what arrived."""
    trees = {"star": wl.star(20), "binary": wl.binary_tree(31), "random40": wl.random_tree(40, 9),
             "star9": wl.star(9, hub=4), "chain": wl.chain(12), **_wide_trees()}
    edges = trees[shape]
    n = int(edges.max()) + 1
    check_tree(n, edges, mode, steps=6, L=2, p_lost=0.25, sums=sums)


def test_received_sums_rows_and_program():
    """relay_set_received_sums: one sum row per wide node (ascending id), one
    more slot per wide node, and nothing changes on a tree without one."""
    star = wl.star(64)
    h = rs.relay_create(64, 8, star)
    assert rs.relay_message_rows(h) == 126
    slots_off = rs.relay_program(h)[0]
    rs.relay_set_received_sums(h, True)
    assert rs.relay_message_rows(h) == 127
    _, _, node, _ = rs.relay_program(h)
    assert node[0][11] == 0 and node[0][10] >= 0 and (node[1:, 10:] == -1).all()
    assert rs.relay_program(h)[0] == slots_off + 1
    rs.relay_set_received_sums(h, False)
    assert rs.relay_message_rows(h) == 126 and rs.relay_program(h)[0] == slots_off
    twin = _wide_trees()["chain3"]
    h = rs.relay_create(23, 8, twin)
    rs.relay_set_received_sums(h, True)
    _, _, node, _ = rs.relay_program(h)
    assert rs.relay_message_rows(h) == 44 + 3
    assert [int(node[i][11]) for i in (0, 2, 4)] == [0, 1, 2]
    for tree in (wl.chain(40), wl.binary_tree(40), wl.torus_spanning_tree(8, 8, 0)):
        n = int(tree.max()) + 1
        a, b = rs.relay_create(n, 8, tree), rs.relay_create(n, 8, tree)
        rs.relay_set_received_sums(b, True)
        assert rs.relay_message_rows(b) == 2 * (n - 1)
        pa, pb = rs.relay_program(a), rs.relay_program(b)
        assert pa[0] == pb[0] and np.array_equal(pa[1], pb[1]) and np.array_equal(pa[2], pb[2])
    lib = ctypes.CDLL(rs.library_path())
    lib.relay_set_received_sums.argtypes = [ctypes.c_void_p, ctypes.c_int32]
    assert lib.relay_set_received_sums(h.raw, 2) == rs.RELAY_EINVAL


def _rebuild_orders(h, n):
    """Per worker: the incoming edges in the order the walk adds them (its
    DFS parent's at its own visit, then each child's at that child's visit),
    derived from the visit order and the parents alone; and the program's
    rebuild-order table, which the node-parallel kernel follows."""
    _, order, node, pos = rs.relay_program(h)
    src, dst = rs.relay_edges(h)
    edge = {(int(a), int(b)): e for e, (a, b) in enumerate(zip(src, dst))}
    walk = {i: [] for i in range(n)}
    for i in order:
        par = node[i][7]
        if par >= 0:
            walk[i].append(edge[(int(par), int(i))])   # the parent's message, at i's visit
            walk[par].append(edge[(int(i), int(par))])  # i's message joins the parent's sum
    table = {i: [int(pos[node[i][1] + k][3]) for k in range(node[i][0])] for i in range(n)}
    return walk, table


def _trees_for_orders():
    out = [(n, e) for n in range(1, 7) for e in tu.all_trees(n)]
    out += [(64, wl.star(64)), (64, wl.torus_spanning_tree(8, 8, 0)), (40, wl.random_tree(40, 1)),
            (32, wl.binary_tree(32)), (16, wl.double_binary_trees(16)[1]), (256, wl.chain(256))]
    return out


def test_rebuild_order_table_follows_the_walk():
    """For every tree up to 6 nodes and the workload trees, the table lists
    each worker's incoming edges exactly once, in the walk's order; adding
    float32 messages in that order reproduces the walk's sums bit for bit."""
    rng = np.random.default_rng(3)
    for n, edges in _trees_for_orders():
        edges = np.asarray(edges, np.int32).reshape(-1, 2)
        h = rs.relay_create(n, 4, edges)
        walk, table = _rebuild_orders(h, n)
        src, dst = rs.relay_edges(h)
        E = 2 * (n - 1)
        m = rng.normal(size=(E, 8)).astype(np.float32)
        base = rng.normal(size=(n, 8)).astype(np.float32)
        for i in range(n):
            assert table[i] == walk[i], (n, i, table[i], walk[i])
            assert sorted(table[i]) == sorted(e for e in range(E) if dst[e] == i)
            a = base[i].copy()
            b = base[i].copy()
            for e in walk[i]:
                a = a + m[e]
            for e in table[i]:
                b = b + m[e]
            assert np.array_equal(a, b)


def test_slot_counts_of_workload_trees():
    """The walk keeps the shared-memory footprint small: O(1) on chains,
    O(depth) on balanced trees, the hub degree on a star."""
    def slots(edges):
        n = int(edges.max()) + 1
        return rs.relay_program(rs.relay_create(n, 4, edges))[0]
    assert slots(wl.chain(64)) <= 3
    assert slots(wl.binary_tree(64)) <= 14
    assert slots(wl.binary_tree(32)) <= 12
    assert slots(wl.star(64)) <= 3

    def slots_with_sums(edges):
        n = int(edges.max()) + 1
        h = rs.relay_create(n, 4, edges)
        rs.relay_set_received_sums(h, True)
        return rs.relay_program(h)[0]
    assert slots_with_sums(wl.star(64)) <= 4
    assert slots(wl.torus_spanning_tree(8, 8, 0)) <= 20


# ------------------------------------------------------------ ABI surface

def _declared_functions():
    import os
    hdr = os.path.join(rs_build.INCLUDE, "relaysum.h")
    text = open(hdr).read()
    return sorted(set(re.findall(r"\b(relay_[a-z_]+)\s*\(", text)))


def test_library_exports_every_declared_symbol():
    lib = ctypes.CDLL(rs.library_path())
    names = _declared_functions()
    assert "relay_step" in names and "relay_create" in names and len(names) >= 15
    for name in names:
        assert hasattr(lib, name), name


@pytest.mark.parametrize("edges,n,status", [
    ([(0, 1), (1, 2), (2, 0)], 3, rs.RELAY_ENOTTREE),
    ([(0, 1), (0, 1)], 3, rs.RELAY_ENOTTREE),
    ([(0, 0)], 2, rs.RELAY_ENOTTREE),
    ([(0, 1), (1, 5)], 3, rs.RELAY_ENOTTREE),
    ([(0, 1)], 3, rs.RELAY_ENOTTREE),
    ([], 0, rs.RELAY_EINVAL),
])
def test_create_rejects_bad_trees(edges, n, status):
    with pytest.raises(rs.RelayError) as e:
        rs.relay_create(n, 8, edges)
    assert e.value.status == status


def test_create_limits_and_layout():
    with pytest.raises(rs.RelayError) as e:
        rs.relay_create(rs.RELAY_MAX_N + 1, 8, wl.chain(rs.RELAY_MAX_N + 1))
    assert e.value.status == rs.RELAY_EUNSUPPORTED
    with pytest.raises(rs.RelayError):
        rs.relay_create(2, -1, [(0, 1)])
    h = rs.relay_create(rs.RELAY_MAX_N, 5, wl.star(rs.RELAY_MAX_N))
    assert rs.relay_num_edges(h) == 2 * (rs.RELAY_MAX_N - 1)
    for d, ld in ((0, 0), (1, 32), (32, 32), (33, 64), (272_474, 272_480)):
        assert rs.relay_ld(rs.relay_create(2, d, [(0, 1)])) == ld
    src, dst = rs.relay_edges(rs.relay_create(4, 8, [(2, 0), (0, 1), (1, 3)]))
    assert list(zip(src, dst)) == tu.directed([(2, 0), (0, 1), (1, 3)])
    h = rs.relay_create(3, 8, [(0, 1), (1, 2)])
    with pytest.raises(rs.RelayError):
        rs.relay_set_rebuild_mode(h, 2)
    for k in (rs.RELAY_KERNEL_WALK, rs.RELAY_KERNEL_NODES):
        rs.relay_set_kernel(h, k)
        assert rs.relay_get_kernel(h) == k
    rs.relay_set_kernel(h, rs.RELAY_KERNEL_AUTO)
    assert rs.relay_get_kernel(h) in (rs.RELAY_KERNEL_WALK, rs.RELAY_KERNEL_NODES)
    for k in (-1, 3):
        with pytest.raises(rs.RelayError) as e:
            rs.relay_set_kernel(h, k)
        assert e.value.status == rs.RELAY_EINVAL
    # relay_steps: the multi-step kernel unless the walk is forced or (AUTO) a node is wide
    for tree, auto in ((wl.chain(8), rs.RELAY_KERNEL_FUSED), (wl.binary_tree(8), rs.RELAY_KERNEL_FUSED),
                       (wl.star(8), rs.RELAY_KERNEL_WALK)):
        hs = rs.relay_create(8, 1 << 24, tree)
        assert rs.relay_get_steps_kernel(hs) == auto
        rs.relay_set_kernel(hs, rs.RELAY_KERNEL_NODES)
        assert rs.relay_get_steps_kernel(hs) == rs.RELAY_KERNEL_FUSED
        rs.relay_set_kernel(hs, rs.RELAY_KERNEL_WALK)
        assert rs.relay_get_steps_kernel(hs) == rs.RELAY_KERNEL_WALK
    with pytest.raises(rs.RelayError):
        rs.relay_set_coord_offset(h, 6)
    rs.relay_set_coord_offset(h, 8)


def test_nbar_host_helper_matches_closed_form():
    edges = wl.binary_tree(7)
    h = rs.relay_create(7, 4, edges)
    counts = np.zeros(12, dtype=np.int32)
    oracle.run(7, edges, np.zeros((7, 0)), np.zeros((7, 0)), np.zeros((12, 0)), counts, 0, 0, 0,
               0, 10, 0)
    assert np.array_equal(rs.relay_nbar(h, counts), np.full(7, 7))


def test_step_rejects_bad_arguments_before_any_launch():
    """Argument checks run on the host before anything touches a device, so
    they are testable without a GPU (the pointers below are never used)."""
    h = rs.relay_create(3, 64, wl.chain(3))
    lib = ctypes.CDLL(rs.library_path())
    lib.relay_step.argtypes = [ctypes.c_void_p] * 5 + [ctypes.c_float, ctypes.c_uint64,
                                                       ctypes.c_int64, ctypes.c_void_p]
    fake = 0x10000
    # no objective bound yet
    assert lib.relay_step(h.raw, fake, fake * 2, fake * 3, fake * 4, 0.1, 0, 0, None) == rs.RELAY_EINVAL
    lib.relay_set_objective.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_float]
    assert lib.relay_set_objective(h.raw, fake, 0.1) == rs.RELAY_OK
    assert lib.relay_set_objective(h.raw, fake + 4, 0.1) == rs.RELAY_EINVAL  # misaligned
    assert lib.relay_set_objective(h.raw, fake, -1.0) == rs.RELAY_EINVAL
    big = 1 << 30
    # msg_in == msg_out, negative step, non-finite lr, overlapping x/messages
    assert lib.relay_step(h.raw, fake, big, big, fake, 0.1, 0, 0, None) == rs.RELAY_EINVAL
    assert lib.relay_step(h.raw, fake, big, 2 * big, fake, 0.1, 0, -1, None) == rs.RELAY_EINVAL
    assert lib.relay_step(h.raw, fake, big, 2 * big, fake, float("nan"), 0, 0, None) == rs.RELAY_EINVAL
    assert lib.relay_step(h.raw, fake, fake + 256, 2 * big, fake, 0.1, 0, 0, None) == rs.RELAY_EINVAL
    assert lib.relay_step(h.raw, fake, big, 2 * big, fake, 0.1, 0, 1 << 32, None) == rs.RELAY_EINVAL
    # relay_steps: the same checks, plus k >= 0 and t0 + k <= 2^32
    lib.relay_steps.argtypes = [ctypes.c_void_p] * 5 + [ctypes.c_float, ctypes.c_uint64, ctypes.c_int64,
                                                        ctypes.c_int64, ctypes.c_void_p]
    assert lib.relay_steps(h.raw, fake, big, big, fake, 0.1, 0, 0, 1, None) == rs.RELAY_EINVAL
    assert lib.relay_steps(h.raw, fake, big, 2 * big, fake, 0.1, 0, -1, 1, None) == rs.RELAY_EINVAL
    assert lib.relay_steps(h.raw, fake, big, 2 * big, fake, float("inf"), 0, 0, 1, None) == rs.RELAY_EINVAL
    assert lib.relay_steps(h.raw, fake, big, 2 * big, fake, 0.1, 0, 0, -1, None) == rs.RELAY_EINVAL
    assert lib.relay_steps(h.raw, fake, big, 2 * big, fake, 0.1, 0, 5, (1 << 32) - 4, None) == rs.RELAY_EINVAL
    assert lib.relay_steps(h.raw, fake, big, 2 * big, fake, 0.1, 0, 0, 0, None) == rs.RELAY_OK  # nothing to do


def test_binding_fails_loudly_without_the_library(monkeypatch, tmp_path):
    """No CPU fallback: with the shared library absent, the first call raises."""
    from paper_2110_04175_gb300 import _native
    monkeypatch.setattr(_native, "_lib", None)
    monkeypatch.setattr(rs_build, "LIB", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="missing"):
        rs.relay_create(3, 8, wl.chain(3))


def test_step_windows_rejects_bad_arguments_before_any_launch():
    """relay_step_windows checks every window (as relay_step does) and its own
    arguments on the host before anything is enqueued."""
    lib = ctypes.CDLL(rs.library_path())
    vp = ctypes.c_void_p
    lib.relay_step_windows.argtypes = [vp, ctypes.c_int32, vp, vp, vp, vp, ctypes.c_float, ctypes.c_uint64,
                                       ctypes.c_int64, vp]
    a, b = wl.double_binary_trees(8)
    ha, hb = rs.relay_create(8, 64, a), rs.relay_create(8, 64, b)
    lib.relay_set_objective.argtypes = [vp, vp, ctypes.c_float]
    fake = 0x10000
    big = 1 << 30
    arr = ctypes.c_void_p * 2
    hs = arr(ha.raw, hb.raw)
    xs, mi, mo, cs = arr(fake, fake + 512), arr(big, big + 512), arr(2 * big, 2 * big + 512), arr(fake * 4, fake * 5)
    # no objective bound on either window
    assert lib.relay_step_windows(hs, 2, xs, mi, mo, cs, 0.1, 0, 0, None) == rs.RELAY_EINVAL
    assert lib.relay_set_objective(ha.raw, fake, 0.1) == rs.RELAY_OK
    assert lib.relay_step_windows(hs, 2, xs, mi, mo, cs, 0.1, 0, 0, None) == rs.RELAY_EINVAL  # window 1
    assert lib.relay_set_objective(hb.raw, fake, 0.1) == rs.RELAY_OK
    for count in (0, 3):
        assert lib.relay_step_windows(hs, count, xs, mi, mo, cs, 0.1, 0, 0, None) == rs.RELAY_EINVAL
    assert lib.relay_step_windows(arr(ha.raw, ha.raw), 2, xs, mi, mo, cs, 0.1, 0, 0, None) == rs.RELAY_EINVAL
    assert lib.relay_step_windows(hs, 2, None, mi, mo, cs, 0.1, 0, 0, None) == rs.RELAY_EINVAL
    assert lib.relay_step_windows(hs, 2, xs, mi, mo, cs, 0.1, 0, -1, None) == rs.RELAY_EINVAL
    assert lib.relay_step_windows(hs, 2, xs, mi, arr(big, 2 * big), cs, 0.1, 0, 0, None) == rs.RELAY_EINVAL
