"""Seeded synthetic inputs for RelaySum runs: trees, mixture weights, workloads.

This module holds input generation only -- none of the method's arithmetic.
Both the CUDA path and the CPU oracle receive what it produces (edge lists,
mixture matrices, scalar hyper-parameters); it imports neither of them.

Workload recipe (stand-ins for the paper's trained models, which are not
used): identity-Hessian heterogeneous quadratics f_i(x) = 1/2 ||x - mu_i||^2
with additive normal gradient noise, on the paper's worker counts (16 workers
in Section 5.2, 16/32/64 in the scaling appendix), topologies (chain as the
spanning tree of a ring, balanced binary trees, the star of the appendix "Star
topology", a random spanning tree as a Spanning-Tree-Protocol stand-in) and
flat parameter vectors of the sizes of its model families (ResNet-20 272,474;
VGG-11 9,231,114; BERT-base 1.1e8).
"""
from __future__ import annotations

import dataclasses

import numpy as np

# --------------------------------------------------------------------- trees


def chain(n: int) -> np.ndarray:
    """Path 0 - 1 - ... - n-1 (the spanning tree of a ring)."""
    return np.array([(i, i + 1) for i in range(n - 1)], dtype=np.int32).reshape(-1, 2)


def binary_tree(n: int) -> np.ndarray:
    """Balanced binary tree in heap order: parent(i) = (i - 1) // 2."""
    return np.array([((i - 1) // 2, i) for i in range(1, n)], dtype=np.int32).reshape(-1, 2)


def inorder_binary_tree(n: int) -> np.ndarray:
    """Binary tree on 0..n-1 in in-order labelling: rank r has label v = r + 1
    in the complete binary tree whose node v sits at height ctz(v); its parent
    is the nearest ancestor with a label <= n.  Every even rank is a leaf and
    every odd rank has a child, so each node has at most three edges."""
    if n <= 1:
        return np.zeros((0, 2), dtype=np.int32)
    top = 1 << (n.bit_length() - 1)          # root label: largest power of two <= n
    edges = []
    for v in range(1, n + 1):
        if v == top:
            continue
        p = v
        while True:
            h = (p & -p).bit_length() - 1    # height of p
            up, down = p + (1 << h), p - (1 << h)
            p = up if (up >> (h + 1)) & 1 else down   # the neighbour label with ctz = h + 1
            if p <= n:
                break
        edges.append((min(v, p) - 1, max(v, p) - 1))
    return np.array(sorted(edges), dtype=np.int32)


def double_binary_trees(n: int):
    """The two complementary trees of Section 3 ("Spanning trees"): tree A is
    the in-order binary tree, tree B its mirror image r -> n-1-r (n even) or
    its shift r -> r+1 mod n (n odd), so that the internal nodes of one tree
    are leaves of the other."""
    a = inorder_binary_tree(n)
    if n % 2 == 0:
        b = (n - 1) - a
    else:
        b = (a + 1) % n
    b = np.sort(b, axis=1)
    return a, np.array(sorted(map(tuple, b)), dtype=np.int32).reshape(-1, 2)


def star(n: int, hub: int = 0) -> np.ndarray:
    """Star: the hub is connected to every other worker."""
    return np.array([(hub, i) for i in range(n) if i != hub], dtype=np.int32).reshape(-1, 2)


def torus_spanning_tree(rows: int, cols: int, seed: int = 0) -> np.ndarray:
    """Uniform random spanning tree of the rows x cols torus grid (Wilson's
    loop-erased random walks, root 0, nodes added in id order).

    Node (r, c) has id r * cols + c; its neighbours are taken in the order
    up, down, left, right (with wrap-around).
    """
    n = rows * cols
    rng = np.random.Generator(np.random.PCG64(seed))

    def nbrs(u: int):
        r, c = divmod(u, cols)
        return [((r - 1) % rows) * cols + c, ((r + 1) % rows) * cols + c,
                r * cols + (c - 1) % cols, r * cols + (c + 1) % cols]

    in_tree = [False] * n
    nxt = [-1] * n
    in_tree[0] = True
    for start in range(n):
        u = start
        while not in_tree[u]:
            nb = nbrs(u)
            nxt[u] = nb[int(rng.integers(0, len(nb)))]
            u = nxt[u]
        u = start
        while not in_tree[u]:
            in_tree[u] = True
            u = nxt[u]
    edges = sorted((min(u, nxt[u]), max(u, nxt[u])) for u in range(1, n))
    return np.array(edges, dtype=np.int32).reshape(-1, 2)


def random_tree(n: int, seed: int = 0) -> np.ndarray:
    """Random labelled tree from a uniformly drawn Pruefer sequence."""
    if n <= 1:
        return np.zeros((0, 2), dtype=np.int32)
    rng = np.random.Generator(np.random.PCG64(seed))
    seq = [int(v) for v in rng.integers(0, n, size=n - 2)]
    return np.array(pruefer_to_edges(n, seq), dtype=np.int32).reshape(-1, 2)


def pruefer_to_edges(n: int, seq) -> list:
    """Decodes a Pruefer sequence of length n-2 into the n-1 tree edges."""
    degree = [1] * n
    for v in seq:
        degree[v] += 1
    edges = []
    for v in seq:
        leaf = min(i for i in range(n) if degree[i] == 1)
        edges.append((min(leaf, v), max(leaf, v)))
        degree[leaf] -= 1
        degree[v] -= 1
    rest = [i for i in range(n) if degree[i] == 1]
    if n >= 2:
        edges.append((rest[0], rest[1]))
    return edges


# ------------------------------------------------------------ mixture weights


def identity_mix(n: int) -> np.ndarray:
    """mu_i = scale * N_i: one independent Gaussian centre per worker."""
    return np.eye(n, dtype=np.float32)


def dirichlet_mix(n: int, K: int, alpha: float, seed: int = 0) -> np.ndarray:
    """mu_i = sum_k w_ik C_k with w_i ~ Dirichlet(alpha * 1_K)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    return rng.dirichlet(alpha * np.ones(K), size=n).astype(np.float32)


# ------------------------------------------------------------------ workloads


@dataclasses.dataclass
class Workload:
    name: str
    n: int
    edges: np.ndarray      # (n-1, 2) int32 undirected tree edges, or a list of
                           # trees splitting the coordinates (double binary trees)
    d: int                 # parameters per worker
    mix: np.ndarray        # (n, K) float32 mixture of Gaussian centres
    mu_scale: float        # mu_i = mu_scale * sum_k mix[i, k] N_k
    sigma: float           # gradient noise standard deviation
    lr: float              # learning rate gamma
    x0_std: float          # x^0 = x0_std * N (shared by all workers)
    steps: int
    seed: int = 0          # Philox key of the noise and of x^0
    mu_seed: int = 0       # Philox key of the centres
    mode: int = 1          # 0: Alg. 1 rebuild, 1: robust rebuild

    @property
    def E(self) -> int:
        return 2 * (self.n - 1)

    def bytes_per_step(self) -> int:
        """Algorithmic HBM bytes of one step: read x (n d) and m^{t-1} (E d),
        write m^t (E d) and x (n d), all fp32."""
        return 4 * self.d * (2 * self.n + 2 * self.E)

    def bytes_per_step_with_mu(self) -> int:
        """As bytes_per_step plus the read of the stored centres mu (n d)."""
        return self.bytes_per_step() + 4 * self.d * self.n


def chain8_d4096() -> Workload:
    n = 8
    return Workload("chain8_d4096", n, chain(n), 4096, identity_mix(n), 2.0, 0.1, 0.1, 0.0, 100)


def binary16_resnet20() -> Workload:
    n = 16
    return Workload("binary16_d272474", n, binary_tree(n), 272_474, identity_mix(n), 1.0, 0.05,
                    0.05, 0.1, 500)


def chain16_vgg11() -> Workload:
    n = 16
    return Workload("chain16_d9231114_dirichlet", n, chain(n), 9_231_114,
                    dirichlet_mix(n, 10, 0.1, seed=0), 1.0, 0.05, 0.05, 0.0, 200)


def binary32_bert() -> Workload:
    n = 32
    return Workload("binary32_d110000000", n, binary_tree(n), 110_000_000, identity_mix(n), 1.0,
                    0.01, 0.01, 0.0, 50)


def sweep64(shape: str) -> Workload:
    n = 64
    trees = {"star": star(n), "chain": chain(n), "binary": binary_tree(n),
             "torus": torus_spanning_tree(8, 8, seed=0)}
    return Workload(f"{shape}64_d25000000", n, trees[shape], 25_000_000, identity_mix(n), 1.0,
                    0.05, 0.05, 0.0, 100)


def double16_vgg11() -> Workload:
    """16 workers on double binary trees (Section 3), VGG-11-sized vector: the
    paper's data-centre topology for its 16-worker experiments."""
    n = 16
    return Workload("double16_d9231114", n, list(double_binary_trees(n)), 9_231_114,
                    identity_mix(n), 1.0, 0.05, 0.05, 0.0, 200)


def all_workloads() -> list:
    return [chain8_d4096(), binary16_resnet20(), chain16_vgg11(), binary32_bert()] + [
        sweep64(s) for s in ("star", "chain", "binary", "torus")] + [double16_vgg11()]


def by_name(name: str) -> Workload:
    for w in all_workloads():
        if w.name == name:
            return w
    raise KeyError(name)
