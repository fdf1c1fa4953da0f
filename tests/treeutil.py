"""Small graph helpers for the tests (independent of both the oracle and the
CUDA library): distances, subtrees behind an edge, every labelled tree."""
from __future__ import annotations

import itertools
from collections import defaultdict

from paper_2110_04175_gb300.workloads import pruefer_to_edges


def adjacency(n, edges):
    adj = defaultdict(list)
    for a, b in edges:
        adj[int(a)].append(int(b))
        adj[int(b)].append(int(a))
    return adj


def distances(n, edges):
    """tau[i][j]: hops between i and j (BFS)."""
    adj = adjacency(n, edges)
    tau = []
    for s in range(n):
        d = {s: 0}
        q = [s]
        for u in q:
            for v in adj[u]:
                if v not in d:
                    d[v] = d[u] + 1
                    q.append(v)
        tau.append([d[j] for j in range(n)])
    return tau


def side(n, edges, i, j):
    """T_{i\\j}: the nodes on i's side once the edge {i, j} is removed."""
    adj = adjacency(n, edges)
    seen = {i}
    q = [i]
    for u in q:
        for v in adj[u]:
            if (u, v) == (i, j) or v in seen:
                continue
            seen.add(v)
            q.append(v)
    return seen


def directed(edges):
    """Directed edge e = 2u: edges[u][0] -> edges[u][1]; 2u+1 the reverse."""
    out = []
    for a, b in edges:
        out.append((int(a), int(b)))
        out.append((int(b), int(a)))
    return out


def all_trees(n):
    """Every labelled tree on n nodes (n^(n-2) of them, via Pruefer codes)."""
    if n == 1:
        yield []
        return
    if n == 2:
        yield [(0, 1)]
        return
    for seq in itertools.product(range(n), repeat=n - 2):
        yield pruefer_to_edges(n, seq)


def diameter(n, edges):
    if n == 1:
        return 0
    return max(max(row) for row in distances(n, edges))
