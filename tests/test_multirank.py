"""World-size-2 checks of the multi-GPU host logic on CPU (gloo).

bench.py shards the model vector over ranks by coordinate: rank r owns the
slice starting at shard_offset(r, d) of one longer vector, with no data-path
collective; the job time is the max over ranks.  Here two gloo ranks run the
oracle on their slices and check that the gathered result equals one
unsharded run, and that the max-reduction and barrier behave.
"""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, result_dir):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        from oracle import oracle
        from paper_2110_04175_gb300 import workloads as wl

        # max / min over ranks
        got = bench.reduce_max(float(rank + 1) * 1.5, world)
        assert got == 1.5 * world
        assert bench.reduce_min(float(rank + 1) * 1.5, world) == 1.5
        bench.barrier(world)

        # d-sharding: each rank runs its slice of a longer vector
        w = wl.Workload("bin7", 7, wl.binary_tree(7), 10, wl.identity_mix(7), 1.0, 0.1, 0.1,
                        0.1, 6)
        c0 = bench.shard_offset(rank, w.d)
        st = oracle.State(w.n, w.edges, w.d, c0=c0)
        st.init(w.x0_std, w.seed, w.mix.astype(np.float64), w.mu_scale, w.mu_seed)
        st.advance(w.steps, w.lr, w.sigma, w.seed, w.mode)
        mine = torch.from_numpy(st.x.copy())
        parts = [torch.zeros_like(mine) for _ in range(world)]
        dist.all_gather(parts, mine)
        if rank == 0:
            stride = bench.shard_offset(1, w.d)
            full = oracle.State(w.n, w.edges, stride * world)
            full.init(w.x0_std, w.seed, w.mix.astype(np.float64), w.mu_scale, w.mu_seed)
            full.advance(w.steps, w.lr, w.sigma, w.seed, w.mode)
            for r in range(world):
                want = full.x[:, r * stride: r * stride + w.d]
                assert np.array_equal(parts[r].numpy(), want)
            open(os.path.join(result_dir, "ok"), "w").write("ok")
    finally:
        dist.destroy_process_group()


def test_two_ranks_shard_over_d_and_reduce_max(tmp_path):
    port = _free_port()
    mp.spawn(_worker, args=(2, port, str(tmp_path)), nprocs=2, join=True)
    assert (tmp_path / "ok").exists()


def test_shard_offsets_are_quad_aligned():
    import bench
    for d in (1, 3, 4, 5, 110_000_000, 9_231_114):
        for r in range(8):
            c0 = bench.shard_offset(r, d)
            assert c0 % 4 == 0 and c0 >= r * d
            assert bench.shard_offset(r + 1, d) - c0 >= d


def test_rank_placement_and_backend():
    """One GPU per local rank: rank i on GPU i over NCCL; more ranks than
    GPUs: round robin over them, host collectives over gloo."""
    import bench
    assert [bench.local_device(r, 8) for r in range(8)] == list(range(8))
    assert [bench.local_device(r, 1) for r in range(4)] == [0, 0, 0, 0]
    assert [bench.local_device(r, 2) for r in range(4)] == [0, 1, 0, 1]
    assert bench.process_group_backend(8, 8) == "nccl"
    assert bench.process_group_backend(1, 1) == "nccl"
    assert bench.process_group_backend(2, 1) == "gloo"
    with pytest.raises(RuntimeError):
        bench.local_device(0, 0)


def _oracle_metrics(x: np.ndarray, mu: np.ndarray):
    """Consensus distance 1/(n d) sum_i ||x_i - xbar||^2 and ||xbar - mubar||^2 / d
    of fp64 models x [n][d] and centres mu [n][d], straight from the definition."""
    xbar = x.mean(axis=0)
    mubar = mu.mean(axis=0)
    return float(((x - xbar) ** 2).sum(axis=0).mean() / x.shape[0]), float(((xbar - mubar) ** 2).mean())


def test_slice_metrics_combine_to_the_whole_vector():
    """Per-slice metrics weighted by slice width equal the whole vector's."""
    import bench
    from oracle import oracle
    from paper_2110_04175_gb300 import workloads as wl
    w = wl.Workload("bin9", 9, wl.binary_tree(9), 1000, wl.identity_mix(9), 1.0, 0.1, 0.1, 0.1, 7)
    st = oracle.State(w.n, w.edges, 3 * w.d)
    st.init(w.x0_std, w.seed, w.mix.astype(np.float64), w.mu_scale, w.mu_seed)
    st.advance(w.steps, w.lr, w.sigma, w.seed, w.mode)
    whole = _oracle_metrics(st.x, st.mu)
    cuts = [0, 400, 1004, 3000]  # ragged slices
    parts = [(b - a, *_oracle_metrics(st.x[:, a:b], st.mu[:, a:b])) for a, b in zip(cuts, cuts[1:])]
    got = bench.combine_slice_metrics(parts)
    assert np.allclose(got, whole, rtol=1e-12, atol=0)
    assert whole[0] > 0 and whole[1] > 0


class _SliceRun:
    """Stands in for a RelayRun in bench.sharded_metrics: the metrics of its
    tree windows and their widths."""

    def __init__(self, windows, t):
        self.trees = [type("W", (), {"d": d})() for d, _, _ in windows]
        self._m = torch.tensor([[c, m] for _, c, m in windows], dtype=torch.float64)
        self.t = t

    def metrics(self):
        return self._m


def _metrics_worker(rank, world, port, result_dir):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        windows = [[(300, 0.5, 2.0), (700, 1.5, 1.0)], [(1000, 3.0, 4.0)]][rank]
        got = bench.sharded_metrics(_SliceRun(windows, 12), world)
        want = bench.combine_slice_metrics([(300, 0.5, 2.0), (700, 1.5, 1.0), (1000, 3.0, 4.0)])
        assert got["coordinates"] == 2000 and got["after_steps"] == 12
        assert np.allclose([got["consensus_distance"], got["distance_to_optimum"]], want, rtol=1e-15)
        if rank == 0:
            open(os.path.join(result_dir, "ok"), "w").write("ok")
    finally:
        dist.destroy_process_group()


def test_sharded_metrics_all_reduce_two_ranks(tmp_path):
    port = _free_port()
    mp.spawn(_metrics_worker, args=(2, port, str(tmp_path)), nprocs=2, join=True)
    assert (tmp_path / "ok").exists()
