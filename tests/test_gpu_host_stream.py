"""The host-state step (relay_step_host / relay_steps_host through
HostRelayRun) equals the fully resident run, bit for bit: the models, the
counters, and every message row it copies back -- the rows a later step
reads (all but those arriving at leaves, plus the wide nodes' received sums),
or every row of m^t with full output."""
import ctypes

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


def _edges(shape, n):
    return {"binary": wl.binary_tree(n), "star": wl.star(n), "chain": wl.chain(n), "pair": wl.chain(n)}[shape]


@pytest.mark.parametrize("full_output", [False, True])
@pytest.mark.parametrize("shape,n,d,chunk,buffers", [
    ("binary", 16, 1_000_003, 1 << 18, 3),   # 4 chunks, ragged last one
    ("star", 12, 70_001, 1 << 14, 2),        # wide node, 5 chunks, 2 buffers
    ("chain", 5, 1_000, 1 << 12, 3),         # a single chunk
    ("pair", 2, 5_000, 1 << 12, 2),          # two leaves: no message row is read
])
def test_host_stream_equals_resident_run(shape, n, d, chunk, buffers, full_output):
    edges = _edges(shape, n)
    w = wl.Workload(shape, n, edges, d, wl.identity_mix(n), 1.0, 0.05, 0.05, 0.1, 7)
    dev = rs.RelayRun(n, d, edges, device="cuda:0")
    dev.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
    host = HostRelayRun(n, d, edges, chunk=chunk, buffers=buffers, device="cuda:0", full_output=full_output)
    host.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
    assert torch.equal(host.models(), dev.x[:, :d].cpu())  # x^0 written chunk by chunk
    for _ in range(w.steps):
        dev.step(w.lr, w.seed)
        host.step(w.lr, w.seed)
    host.sync()
    torch.cuda.synchronize()
    assert torch.equal(host.models(), dev.x[:, :d].cpu())
    assert torch.equal(host.counts_h[:dev.E], dev.counts[:dev.E].cpu())
    # the rows a step reads: all but those arriving at a leaf, and the
    # received-sum rows of the wide nodes (the star's hub)
    src, dst = rs.relay_edges(dev.h)
    degree = np.bincount(np.asarray(dst), minlength=n)
    rows = rs.relay_message_rows(dev.h)
    assert host.kept_rows == [e for e in range(dev.E) if degree[dst[e]] > 1] + list(range(dev.E, rows))
    assert rows == dev.E + int((degree > 4).sum())
    got = host.messages()
    if full_output:
        assert torch.equal(got, dev.messages[:dev.E, :d].cpu())
    else:
        kept = [e for e in host.kept_rows if e < dev.E]
        assert torch.equal(got[kept], dev.messages[:dev.E, :d].cpu()[kept])
        dropped = [e for e in range(dev.E) if e not in kept]
        assert torch.isnan(got[dropped]).all()
    if rows > dev.E:  # the sum rows went out and back too
        assert torch.equal(host.msg_h[host.cur][dev.E:rows, :d], dev.messages[dev.E:rows, :d].cpu())
    # the bytes the library reports: x, the rows in / out and the counters
    h2d, d2h = host.bytes_per_step()
    cols = sum((min(host.cw, d - k * host.cw) + 3) // 4 * 4 for k in range(host.nchunks))
    assert h2d == 4 * (cols * (n + len(host.kept_rows)) + dev.E)
    assert d2h == 4 * (cols * (n + (rows if full_output else len(host.kept_rows))) + dev.E)


@pytest.mark.parametrize("shape,n,d,chunk,buffers", [
    ("binary", 16, 1_000_003, 1 << 18, 3),   # 4 chunks, multi-step kernel
    ("star", 12, 70_001, 1 << 14, 2),        # wide node: relay_steps repeats relay_step
    ("chain", 5, 1_000, 1 << 12, 3),         # a single chunk
    ("pair", 2, 5_000, 1 << 12, 2),          # no message row read
])
def test_host_stream_steps_equal_resident_steps(shape, n, d, chunk, buffers):
    """HostRelayRun.steps(k): one relay_steps call per chunk visit, every chunk
    starting from the same counters, mixed with single steps, equals the
    resident run step by step on x, the counters and the rows copied back."""
    edges = _edges(shape, n)
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
        kept = [e for e in host.kept_rows if e < dev.E]
        assert torch.equal(host.messages()[kept], dev.messages[:dev.E, :d].cpu()[kept]), k


def test_host_step_rejects_what_it_cannot_stream():
    """relay_step_host takes page-locked host arrays and a handle whose inputs
    all live in them: pageable or device memory, stored centres and an
    optimiser with state are refused before anything is enqueued."""
    n, d = 6, 4096
    host = HostRelayRun(n, d, wl.chain(n), chunk=1024, device="cuda:0")
    host.init(0.1, 1, wl.identity_mix(n), 1.0, 2, 0.1)
    lib = ctypes.CDLL(rs.library_path())
    vp = ctypes.c_void_p
    lib.relay_step_host.argtypes = [vp, vp, vp, vp, vp, ctypes.c_float, ctypes.c_uint64, ctypes.c_int64, vp]
    pageable = np.zeros((n, host.ld), np.float32)
    args = [host.msg_h[0].data_ptr(), host.msg_h[1].data_ptr(), host.counts_h.data_ptr()]
    x = host.x_h.data_ptr()
    assert lib.relay_step_host(host.plan.raw, pageable.ctypes.data, *args, 0.1, 1, 0, None) == rs.RELAY_EINVAL
    dev_x = torch.zeros(n, host.ld, device="cuda:0")
    assert lib.relay_step_host(host.plan.raw, dev_x.data_ptr(), *args, 0.1, 1, 0, None) == rs.RELAY_EINVAL
    assert lib.relay_step_host(host.plan.raw, x, *args, float("nan"), 1, 0, None) == rs.RELAY_EINVAL
    assert lib.relay_step_host(host.plan.raw, x, *args, 0.1, 1, -1, None) == rs.RELAY_EINVAL
    mu = torch.zeros(n, host.ld, device="cuda:0")
    rs.relay_set_objective(host.h, mu, 0.1)
    assert lib.relay_step_host(host.plan.raw, x, *args, 0.1, 1, 0, None) == rs.RELAY_EUNSUPPORTED
    rs.relay_set_objective_generated(host.h, wl.identity_mix(n), n, 1.0, 2, 0.1)
    state = torch.zeros(n, host.ld, device="cuda:0")
    rs.relay_set_local_optimizer(host.h, rs.RELAY_OPT_NESTEROV, 0.9, 0.0, 0.0, state, None)
    assert lib.relay_step_host(host.plan.raw, x, *args, 0.1, 1, 0, None) == rs.RELAY_EUNSUPPORTED
    rs.relay_set_local_optimizer(host.h, rs.RELAY_OPT_SGD)
    assert lib.relay_step_host(host.plan.raw, x, *args, 0.1, 1, 0, None) == rs.RELAY_OK
    torch.cuda.synchronize()
    # the staging must be large enough
    small = torch.empty(rs.relay_host_staging_bytes(host.h, 1024, 3) - 256, dtype=torch.uint8, device="cuda:0")
    with pytest.raises(rs.RelayError):
        rs.relay_host_plan_create(host.h, 1024, 3, small)
