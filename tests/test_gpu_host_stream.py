"""The host-state streaming mode equals the fully resident run, bit for bit,
on everything it keeps: the models, the counters and every message row that
a later step reads (all but the rows arriving at leaves)."""
import numpy as np
import pytest
import torch

import paper_2110_04175_gb300 as rs
from paper_2110_04175_gb300 import workloads as wl
from paper_2110_04175_gb300.host_stream import HostRelayRun

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


@pytest.mark.parametrize("shape,n,d,chunk,buffers", [
    ("binary", 16, 1_000_003, 1 << 18, 3),   # 4 chunks, ragged last one
    ("star", 12, 70_001, 1 << 14, 2),        # wide node, 5 chunks, 2 buffers
    ("chain", 5, 1_000, 1 << 12, 3),         # a single chunk
    ("pair", 2, 5_000, 1 << 12, 2),          # two leaves: no message row is kept
])
def test_host_stream_equals_resident_run(shape, n, d, chunk, buffers):
    edges = {"binary": wl.binary_tree(n), "star": wl.star(n), "chain": wl.chain(n),
             "pair": wl.chain(n)}[shape]
    w = wl.Workload(shape, n, edges, d, wl.identity_mix(n), 1.0, 0.05, 0.05, 0.1, 7)
    dev = rs.RelayRun(n, d, edges, device="cuda:0")
    dev.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
    host = HostRelayRun(n, d, edges, chunk=chunk, buffers=buffers, device="cuda:0")
    host.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
    for _ in range(w.steps):
        dev.step(w.lr, w.seed)
        host.step(w.lr, w.seed)
    host.sync()
    torch.cuda.synchronize()
    assert torch.equal(host.models(), dev.x[:, :d].cpu())
    assert torch.equal(host.counts_h[:dev.E], dev.counts[:dev.E].cpu())
    # the kept rows are exactly those whose receiver is not a leaf
    src, dst = rs.relay_edges(dev.h)
    degree = np.bincount(np.asarray(dst), minlength=n)
    assert host.kept_rows == [e for e in range(dev.E) if degree[dst[e]] > 1]
    got = host.messages()
    kept = host.kept_rows
    assert torch.equal(got[kept], dev.messages[:dev.E, :d].cpu()[kept])
    dropped = [e for e in range(dev.E) if e not in kept]
    assert torch.isnan(got[dropped]).all()


@pytest.mark.parametrize("shape,n,d,chunk,buffers", [
    ("binary", 16, 1_000_003, 1 << 18, 3),   # 4 chunks, multi-step kernel
    ("star", 12, 70_001, 1 << 14, 2),        # wide node: relay_steps repeats relay_step
    ("chain", 5, 1_000, 1 << 12, 3),         # a single chunk
    ("pair", 2, 5_000, 1 << 12, 2),          # no message row kept
])
def test_host_stream_steps_equal_resident_steps(shape, n, d, chunk, buffers):
    """HostRelayRun.steps(k): one relay_steps call per chunk visit, every chunk
    starting from the same counters, mixed with single steps, equals the
    resident run step by step on x, the counters and the kept message rows."""
    edges = {"binary": wl.binary_tree(n), "star": wl.star(n), "chain": wl.chain(n),
             "pair": wl.chain(n)}[shape]
    w = wl.Workload(shape, n, edges, d, wl.identity_mix(n), 1.0, 0.05, 0.05, 0.1, 7)
    dev = rs.RelayRun(n, d, edges, device="cuda:0")
    dev.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
    host = HostRelayRun(n, d, edges, chunk=chunk, buffers=buffers, device="cuda:0")
    host.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
    for k in (1, 2, 64, 65, 3, 0):
        for _ in range(k):
            dev.step(w.lr, w.seed)
        host.steps(k, w.lr, w.seed)
        host.step(w.lr, w.seed)
        dev.step(w.lr, w.seed)
        host.sync()
        torch.cuda.synchronize()
        assert host.t == dev.t
        assert torch.equal(host.models(), dev.x[:, :d].cpu()), k
        assert torch.equal(host.counts_h[:dev.E], dev.counts[:dev.E].cpu()), k
        kept = host.kept_rows
        assert torch.equal(host.messages()[kept], dev.messages[:dev.E, :d].cpu()[kept]), k
