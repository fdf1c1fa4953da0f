"""Throughput of the RelaySum step (RelaySGD, arXiv 2110.04175, Algorithm 1).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl native|reference]
                    [--workload NAME] [--e2e-steps K2] [--no-cpu-baseline]

A step is one RelaySGD iteration of the whole hot path -- counter update,
local step with Philox gradient noise, every relay message, every rebuild --
over the default workload: 32 workers on a balanced binary tree, d = 1.1e8
fp32 parameters each (a BERT-base-sized flat vector), robust rebuild.  The
per-step working set (82.7 GB moved) is far larger than L2, so no flush is
needed between steps.  Inputs are seeded synthetic quadratics.

Prints one JSON line.  `value` is whole-job steps/s with the state resident
in HBM; `e2e` is the same metric through relay_step_host with the state in
pinned host buffers (copies inside the timed region); `roofline` is the step
kernel's algorithmic HBM bytes per launch over its CUDA-event duration;
`cpu_baseline` times the plain CPU oracle on a bounded coordinate sample,
on every host core (one slice per thread) and on one thread; `metrics` is the
consensus distance and the average model's distance to the optimum after the
timed steps, over every rank's slice.

Multi-GPU (torchrun, one rank per GPU): every rank runs the same workload on
its own d-slice of one longer model vector (coordinates are independent, so
there is no data-path collective; weak scaling; the one collective, after the
timed region, sums the ranks' metrics).  With more local ranks than
visible GPUs the ranks share them round robin and the process group uses
gloo (a functional check of the multi-rank path; such a line is no scaling
figure).  `--impl reference` times the CPU oracle instead (rank 0 only).
"""
from __future__ import annotations

import argparse
import gc
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "RelaySum steps/s and achieved HBM GB/s (fraction of GB300 peak) vs CPU oracle"
DEFAULT_WORKLOAD = "binary32_d110000000"
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 7900.0  # GB300 HBM3e, nominal


# ------------------------------------------------------------ host helpers

def shard_offset(rank: int, d: int) -> int:
    """First absolute coordinate of rank `rank`'s slice (multiple of 4)."""
    return rank * ((d + 3) // 4 * 4)


def reduce_max(value: float, world: int) -> float:
    """Max over ranks (the slowest rank sets the job time)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([value], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def reduce_min(value: float, world: int) -> float:
    """Min over ranks (used for decisions every rank must take alike)."""
    return -reduce_max(-value, world)


def local_device(local: int, n_devices: int) -> int:
    """The GPU of local rank `local`: its own where every local rank has one,
    else round robin over the visible GPUs (the ranks then share them)."""
    if n_devices <= 0:
        raise RuntimeError("bench.py's native arm needs a CUDA device")
    return local % n_devices


def process_group_backend(local_world: int, n_devices: int) -> str:
    """NCCL where every local rank has a GPU of its own; gloo (host
    collectives) where ranks share one, which NCCL refuses.  The path has no
    data-path collective, only the barrier and the max over ranks."""
    return "nccl" if local_world <= n_devices else "gloo"


def combine_slice_metrics(parts) -> tuple:
    """Whole-vector (consensus distance, distance of the average model to the
    optimum) from the metrics of coordinate slices.  relay_metrics gives each
    as a mean over its slice's coordinates (1/(n d) sum_i ||x_i - xbar||^2 and
    ||xbar - mubar||^2 / d), so the whole vector's is the mean of the slices'
    weighted by their widths.  parts: [(d_slice, consensus, distance)]."""
    total = sum(p[0] for p in parts)
    if total <= 0:
        return 0.0, 0.0
    return (sum(p[0] * p[1] for p in parts) / total, sum(p[0] * p[2] for p in parts) / total)


def sharded_metrics(run, world: int) -> dict:
    """The run's metrics over every rank's slice (and tree window): the one
    collective of the d-sharded path, an all-reduce of three doubles, taken
    after the timed region."""
    import torch
    m = run.metrics().cpu().tolist()
    # width-weighted sums over this rank's tree windows, then over the ranks
    sums = [sum(tr.d * m[k][0] for k, tr in enumerate(run.trees)),
            sum(tr.d * m[k][1] for k, tr in enumerate(run.trees)),
            float(sum(tr.d for tr in run.trees))]
    if world > 1:
        import torch.distributed as dist
        dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
        t = torch.tensor(sums, dtype=torch.float64, device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.SUM)
        sums = t.cpu().tolist()
    c, dist_opt = combine_slice_metrics([(sums[2], sums[0] / sums[2], sums[1] / sums[2])] if sums[2] > 0 else [])
    return {"consensus_distance": c, "distance_to_optimum": dist_opt, "after_steps": run.t,
            "coordinates": int(sums[2]),
            "note": "relay_metrics per rank and tree window, combined by slice width"
                    + (" with one all-reduce of 3 doubles after the timed region" if world > 1 else "")}


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def measured_peaks() -> dict:
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return json.load(f)
    except (OSError, ValueError):
        return {}


class ClockSampler:
    """nvidia-smi samples (every 200 ms) of the GPU's clocks and throttle
    reasons while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, bus_id: str | None):
        self.proc = None
        self.file = None
        self.bus_id = bus_id

    def __enter__(self):
        try:
            self.file = tempfile.TemporaryFile(mode="w+")
            cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                   "-lms", "200"]
            if self.bus_id:
                cmd += ["-i", self.bus_id]
            self.proc = subprocess.Popen(cmd, stdout=self.file, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if self.proc is None or self.file is None:
            return None
        self.file.seek(0)
        rows = [r.split(",") for r in self.file.read().strip().splitlines() if r.strip()]
        samples = []
        for r in rows:
            try:
                samples.append({"sm": float(r[1]), "max": float(r[2]), "power": float(r[3]),
                                "hw": r[5].strip(), "hw_thermal": r[6].strip(),
                                "sw_thermal": r[7].strip(), "sw_power": r[8].strip()})
            except (ValueError, IndexError):
                continue
        if not samples:
            return None
        peak_power = max(s["power"] for s in samples)
        loaded = [s for s in samples if s["power"] >= 0.5 * peak_power] or samples
        reasons = set()
        for s in loaded:
            for key, name in (("hw", "hw_slowdown"), ("hw_thermal", "hw_thermal_slowdown"),
                              ("sw_thermal", "sw_thermal_slowdown"), ("sw_power", "sw_power_cap")):
                if s[key].lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(s["sm"] for s in loaded),
                "sm_max_mhz": max(s["max"] for s in samples),
                "reasons": sorted(reasons), "samples": len(samples), "samples_under_load": len(loaded),
                "power_w_max": peak_power}


def bus_id_of(device: int) -> str | None:
    """nvidia-smi's id (its PCI bus id) of the torch device, or None."""
    import torch
    p = torch.cuda.get_device_properties(device)
    want = tuple(getattr(p, k, None) for k in ("pci_domain_id", "pci_bus_id", "pci_device_id"))
    try:
        out = subprocess.run(["nvidia-smi", "--query-gpu=pci.bus_id", "--format=csv,noheader"],
                             capture_output=True, text=True, timeout=30).stdout
    except (OSError, subprocess.SubprocessError):
        return None
    ids = [line.strip() for line in out.splitlines() if line.strip()]
    for bus in ids:
        try:
            dom, b, rest = bus.split(":")
            if (int(dom, 16), int(b, 16), int(rest.split(".")[0], 16)) == want:
                return bus
        except ValueError:
            continue
    return ids[0] if len(ids) == 1 else None


# -------------------------------------------------------------- CPU oracle

def host_threads() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


class OracleSlices:
    """The oracle, as it stands, on `threads` disjoint consecutive coordinate
    slices of workload `w`, advanced concurrently (each thread one slice; the
    ctypes calls release the GIL, so the slices run on separate cores)."""

    def __init__(self, w, length: int, threads: int):
        import numpy as np
        from oracle import oracle
        edges = w.edges[0] if isinstance(w.edges, list) else w.edges  # a sample in the first window
        self.w, self.length, self.threads = w, length, threads
        self.states = [oracle.State(w.n, edges, length, c0=k * length) for k in range(threads)]
        self.pool = None
        if threads > 1:
            from concurrent.futures import ThreadPoolExecutor
            self.pool = ThreadPoolExecutor(threads)
        mix = w.mix.astype(np.float64)
        self._each(lambda st: st.init(w.x0_std, w.seed, mix, w.mu_scale, w.mu_seed))

    def _each(self, fn):
        if self.pool is None:
            fn(self.states[0])
        else:
            list(self.pool.map(fn, self.states))

    def advance(self, steps: int) -> float:
        """Wall-clock seconds for `steps` steps of every slice."""
        w = self.w
        t0 = time.perf_counter()
        self._each(lambda st: st.advance(steps, w.lr, w.sigma, w.seed, w.mode))
        return time.perf_counter() - t0

    def close(self):
        if self.pool is not None:
            self.pool.shutdown()


def oracle_bytes_per_coord(w) -> int:
    """Host bytes one oracle coordinate holds: x, mu, messages and the
    step's temporaries (x^{t+1/2}, new messages), fp64."""
    return 8 * (3 * w.n + 2 * 2 * (w.n - 1))


def oracle_plan(w, threads: int, mem_per_thread: int):
    """(threads, coordinates per thread) for a concurrent oracle sample of
    `w`: at most `mem_per_thread` host bytes per slice, within d."""
    cap = max(4, mem_per_thread // oracle_bytes_per_coord(w))
    threads = max(1, min(threads, w.d // 1024))
    return threads, max(4, min(cap, w.d // threads) // 4 * 4)


def oracle_per_coord(w) -> float:
    """One-thread seconds per coordinate-step of the oracle on `w`."""
    probe = OracleSlices(w, min(4096, max(4, w.d // 4 * 4)), 1)
    probe.advance(1)
    dt = probe.advance(1)
    return dt / probe.length


def oracle_sample(w, seconds: float = 8.0):
    """Times the oracle (as it stands) on bounded coordinate samples of
    workload `w`, scaled to steps/s of the full d: on every host core (one
    slice per thread) and, for reference, on one thread.  The slices are
    small (the oracle's centre fill costs about as much as 25 steps) and
    the step counts fill about `seconds` each at one thread's rate."""
    per_coord = oracle_per_coord(w)
    threads, lt = oracle_plan(w, host_threads(), 96 << 20)
    steps = int(max(2, min(200, round(seconds / (lt * per_coord)))))
    one = OracleSlices(w, lt, 1)
    steps1 = max(1, steps // 2)
    dt1 = one.advance(steps1)
    one.close()
    del one
    many = OracleSlices(w, lt, threads)
    dt = many.advance(steps)
    many.close()
    del many
    return {"value": steps / dt * threads * lt / w.d, "unit": "steps/s", "cores": threads,
            "kind": "oracle", "value_1thread": steps1 / dt1 * lt / w.d,
            "sample": f"{steps} steps of coordinates [0, {threads * lt}) of d = {w.d}, "
                      f"{threads} threads of {lt} coordinates each ({dt:.1f} s), scaled by "
                      f"{threads * lt}/{w.d}; value_1thread: {steps1} steps of [0, {lt}) on one "
                      f"thread ({dt1:.1f} s)"}


def run_reference(args, w, rank: int):
    """The reference arm: the plain CPU oracle on bounded samples of the
    same workload; each step is one oracle step over a coordinate slice per
    host core, run concurrently."""
    if rank != 0:
        return
    per_coord = oracle_per_coord(w)
    budget = 90.0 / max(1, args.steps + args.warmup)  # seconds per step at one thread's rate
    threads, lt = oracle_plan(w, host_threads(), 192 << 20)
    lt = max(4, min(lt, int(budget / per_coord)) // 4 * 4)
    sl = OracleSlices(w, lt, threads)
    if args.warmup:
        sl.advance(args.warmup)
    dt = sl.advance(args.steps)
    sl.close()
    length = threads * lt
    value = args.steps / dt * length / w.d
    sample = (f"each step: one oracle step over coordinates [0, {length}) of d = {w.d}, "
              f"{threads} threads of {lt} coordinates each; steps/s scaled by {length}/{w.d}")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "steps/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": dt / args.steps * 1e3 * w.d / length, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(w, args.gpus, args),
            "cpu_baseline": {"value": value, "unit": "steps/s", "cores": threads, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": "steps/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def l2_bytes(dev) -> int:
    import torch
    return int(getattr(torch.cuda.get_device_properties(dev), "L2_cache_size", 0) or (129 << 20))


def step_bytes(w, args=None) -> int:
    """HBM bytes one step touches: the algorithmic bytes plus the stored mu."""
    stored = args is None or args.objective == "stored"
    return w.bytes_per_step() + (4 * w.d * w.n if stored else 0)


def l2_flush_needed(w, args, dev) -> bool:
    if args.l2_flush != "auto":
        return args.l2_flush == "on"
    return step_bytes(w, args) < 2 * l2_bytes(dev)


def l2_note(w, args, dev=None) -> str:
    mb = step_bytes(w, args) / 1e6
    if args is not None and args.graph:
        return (f"working set {mb:.1f} MB per step; the captured steps run back to back with no "
                f"L2 flush between them (L2-resident where it fits)")
    if dev is not None and args is not None and l2_flush_needed(w, args, dev):
        return (f"working set {mb:.1f} MB per step, under twice the L2: L2 flushed (memset of "
                f"{2 * l2_bytes(dev) / 1e6:.0f} MB) before every timed step, steps timed one by one")
    return f"inputs larger than L2 ({mb / 1e3:.1f} GB moved per step)"


def parallelism_note(gpus: int) -> str:
    if gpus <= 1:
        return "1 GPU"
    note = f"d-sharded over {gpus} rank(s), no collective"
    try:
        import torch
        n_dev = torch.cuda.device_count()
    except Exception:  # noqa: BLE001 - the note is informational
        return note
    local_world = int(os.environ.get("LOCAL_WORLD_SIZE", str(gpus)))
    if 0 < n_dev < local_world:
        note += f"; {local_world} local ranks share {n_dev} GPU(s) (functional check, not a scaling figure)"
    return note


def workload_config(w, gpus: int, args=None, dev=None) -> dict:
    shape = {"binary": "balanced binary tree (heap order)", "chain": "chain", "star": "star",
             "torus": "uniform spanning tree of the 8x8 torus",
             "double": "double binary trees (two complementary trees, half the coordinates each)"}
    kind = next((v for k, v in shape.items() if w.name.startswith(k)), w.name)
    return {"workload": w.name, "n_workers": w.n, "tree": kind, "d": w.d, "directed_edges": w.E,
            "rebuild": "robust (Section 4.4)" if w.mode == 1 else "Algorithm 1",
            "sigma": w.sigma, "lr": w.lr, "objective": "identity-Hessian heterogeneous quadratics",
            "l2": l2_note(w, args, dev),
            "parallelism": parallelism_note(gpus),
            **({"algorithm": args.algorithm, "local_optimizer": args.optimizer,
                "lost_prob": args.lost_prob, "mu": args.objective} if args is not None else {})}


# ------------------------------------------------------------------ native

def make_run(args, w, dev, c0: int):
    """The resident run of workload `w` on `dev`, initialised (RelayRun owns
    the buffers; the library's kernels do all the work)."""
    import paper_2110_04175_gb300 as rs
    optimizer = {"sgd": None, "nesterov": ("nesterov", 0.9),
                 "adam": ("adam", 0.9, 0.999, 1e-8)}[args.optimizer]
    run = rs.RelayRun(w.n, w.d, w.edges, device=dev, mode=w.mode, c0=c0, objective=args.objective,
                      optimizer=optimizer, algorithm=args.algorithm, kernel=args.kernel)
    run.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)
    return run


def make_stepper(args, w, run, stream, rank: int):
    """one_step(ev): one step of `run` on `stream` through the library's step
    call -- relay_step (the step kernel a programmatic dependent of the
    counter kernel), or relay_step_windows for several tree windows --
    bracketed by the CUDA events ev = (start, end) when given."""
    import numpy as np
    import torch

    import paper_2110_04175_gb300 as rs

    lost_rng = np.random.default_rng(1234 + rank)

    def one_step(ev=None):
        torch.cuda.nvtx.range_push(f"relay_step {run.t}")  # a named range per step for profilers
        for tr in run.trees:
            if args.lost_prob > 0:  # messages lost in transit this step (Section 4.4)
                rs.relay_set_lost_messages(tr.h, lost_rng.random(tr.E) < args.lost_prob)
        if ev is not None:
            ev[0].record(stream)
        run.step(w.lr, w.seed, stream)
        if ev is not None:
            ev[1].record(stream)
        torch.cuda.nvtx.range_pop()

    return one_step


def time_steps(args, w, run, one_step, dev, stream, rank: int, world: int, local: int):
    """Times args.steps steps (after the warm-up already run): (total ms,
    max over ranks; the duration of every step; clock summary).  Each step
    is one library call bracketed by two CUDA events on the launching
    stream; its duration is the step kernel's plus whatever of the counter
    kernel the programmatic dependent launch does not overlap."""
    import torch
    # a working set that fits in L2 is evicted before every timed step (a
    # memset of twice the L2), and the steps are then timed one by one
    flush = None
    if l2_flush_needed(w, args, dev):
        flush = torch.empty(2 * l2_bytes(dev), dtype=torch.uint8, device=dev)
    events = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
    torch.cuda.synchronize(dev)
    barrier(world)
    torch.cuda.synchronize(dev)
    with ClockSampler(bus_id_of(local) if rank == 0 else None) as clocks:
        for k in range(args.steps):
            if flush is not None:
                flush.zero_()
            one_step(events[k])
        torch.cuda.synchronize(dev)
    barrier(world)
    torch.cuda.synchronize(dev)
    step_ms = [events[k][0].elapsed_time(events[k][1]) for k in range(args.steps)]
    if flush is None:
        total_ms = events[0][0].elapsed_time(events[-1][1])
    else:
        total_ms = sum(step_ms)
        del flush
    return reduce_max(total_ms, world), step_ms, clocks.summary()


def kernel_name_of(run) -> str:
    import paper_2110_04175_gb300 as rs
    name = ("relay_nodes_kernel" if rs.relay_get_kernel(run.h) == rs.RELAY_KERNEL_NODES
            else "relay_models_kernel")
    T = len(run.trees)
    return name if T == 1 else f"{name} over {T} tree windows in one launch (relay_step_windows)"


def roofline_of(args, w, run, models_ms) -> dict:
    """The step kernel's algorithmic HBM bytes per launch over the mean
    CUDA-event time of the step call that launches it (the step kernel plus
    the part of the one-CTA counter kernel its programmatic dependent launch
    does not overlap: an upper bound on the kernel's own time), against the
    measured copy bandwidth."""
    peaks = measured_peaks()
    peak = peaks.get("hbm_gbs")
    peak_src = "measured" if peak else "fallback"
    peak = peak or FALLBACK_HBM_GBS
    mean_models_ms = statistics.mean(models_ms)
    state_rows = {"sgd": 0, "nesterov": 2, "adam": 4}[args.optimizer]  # optimiser state read+write
    alg_bytes = w.bytes_per_step() + 4 * w.d * w.n * state_rows
    source = run.objective_source
    mu_rows = {"stored": w.n, "generated": 0}[source]
    moved = alg_bytes + 4 * w.d * mu_rows  # the design also reads the stored mu
    achieved = alg_bytes / (mean_models_ms / 1e3) / 1e9
    name = kernel_name_of(run)
    base = name.split(" ")[0]
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4),
                "traffic": traffic_per_launch(w, source, base, args.optimizer),
                "kernel": name, "peak_source": peak_src,
                "algorithmic_bytes_per_launch": alg_bytes,
                "algorithmic_bytes_rule": "4 d (2n + 2E) [+ 4 d n x optimiser-state rows]",
                "objective": source,
                "design_bytes_per_launch": moved,
                "achieved_design_bytes": round(moved / (mean_models_ms / 1e3) / 1e9, 1),
                "launch_ms_mean": round(mean_models_ms, 4),
                "launch_ms_min": round(min(models_ms), 4),
                "timed": "each relay_step call between two CUDA events on its stream (counter kernel, then "
                         "the step kernel as its programmatic dependent)",
                "nominal_peak": NOMINAL_HBM_GBS,
                "frac_of_nominal": round(achieved / NOMINAL_HBM_GBS, 4)}
    if roofline["traffic"]:
        # the ncu DRAM bytes of one launch over this run's mean launch time
        roofline["dram_gbs"] = round(roofline["traffic"] / (mean_models_ms / 1e3) / 1e9, 1)
        roofline["dram_frac"] = round(roofline["dram_gbs"] / peak, 4)
    return roofline


def run_native(args, w, rank: int, world: int):
    import torch

    local = local_device(int(os.environ.get("LOCAL_RANK", "0")), torch.cuda.device_count())
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    c0 = shard_offset(rank, w.d)
    run = make_run(args, w, dev, c0)
    one_step = make_stepper(args, w, run, stream, rank)
    T = len(run.trees)
    for _ in range(args.warmup):
        one_step()
    if args.graph:
        return run_graphed(args, w, run, dev, stream, rank, world)
    total_ms, models_ms, clocks = time_steps(args, w, run, one_step, dev, stream, rank, world, local)
    steps_per_s = world * args.steps / (total_ms / 1e3)
    roofline = roofline_of(args, w, run, models_ms) if rank == 0 else None
    alg_bytes = w.bytes_per_step()
    metrics = sharded_metrics(run, world)

    # several steps per call, on the resident run (before run_e2e frees it)
    fused = run_fused(args, w, run, dev, stream, world) if args.fused_steps > 0 else None
    # end to end: state in pinned host memory, copied in and out every step
    e2e = None
    if args.e2e_steps > 0:
        e2e = run_e2e(args, w, run, dev, stream, world)
    del run, one_step
    gc.collect()
    torch.cuda.empty_cache()
    # the other HBM-bound workloads, each timed like the headline
    per_workload = None
    if args.per_workload and args.d is None:
        per_workload = run_per_workload(args, w, dev, stream, rank, world, local)

    if rank != 0:
        return
    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        cpu = oracle_sample(w)
    line = {"metric": METRIC, "value": round(steps_per_s, 4), "unit": "steps/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(total_ms / args.steps, 4), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": workload_config(w, world, args, dev), "roofline": roofline, "cpu_baseline": cpu,
            "e2e": e2e, "gpu_launches": world * 2 * T * args.steps, "clocks": clocks,
            "hbm_gbs_step": round(alg_bytes * world * args.steps / (total_ms / 1e3) / 1e9, 1),
            "fused_steps": fused, "per_workload": per_workload, "metrics": metrics}
    print(json.dumps(line), flush=True)


PER_WORKLOAD = ["chain16_d9231114_dirichlet", "star64_d25000000", "chain64_d25000000",
                "binary64_d25000000", "torus64_d25000000", "double16_d9231114"]


def run_per_workload(args, head, dev, stream, rank: int, world: int, local: int) -> list:
    """Each of the other HBM-bound workloads (the 16-worker VGG-11-sized chain
    with Dirichlet centres; the four 64-worker trees at d = 2.5e7; the double
    binary trees), timed as the headline is: a fresh resident run, the same
    warm-up and step count, CUDA events on the launching stream, the clocks
    sampled meanwhile.  Each run's buffers are freed before the next."""
    import torch

    from paper_2110_04175_gb300 import workloads as wl

    out = []
    for name in PER_WORKLOAD:
        if name == head.name:
            continue
        w = wl.by_name(name)
        run = make_run(args, w, dev, shard_offset(rank, w.d))
        one_step = make_stepper(args, w, run, stream, rank)
        for _ in range(args.warmup):
            one_step()
        total_ms, models_ms, clocks = time_steps(args, w, run, one_step, dev, stream, rank, world, local)
        if rank == 0:
            cfg = workload_config(w, world, args, dev)
            out.append({"workload": name, "value": round(world * args.steps / (total_ms / 1e3), 4),
                        "unit": "steps/s", "ms_per_step": round(total_ms / args.steps, 4),
                        "n_workers": w.n, "tree": cfg["tree"], "d": w.d, "steps": args.steps,
                        "warmup": args.warmup, "l2": cfg["l2"],
                        "roofline": roofline_of(args, w, run, models_ms), "clocks": clocks,
                        "gpu_launches": world * 2 * len(run.trees) * args.steps})
        del run, one_step
        gc.collect()
        torch.cuda.empty_cache()
    return out


def run_fused(args, w, run, dev, stream, world: int) -> dict:
    """The same workload through relay_steps: K steps per call, the state
    kept on chip between them (the result equals K relay_step calls bit for
    bit).  Its HBM traffic is one read and one write of the state per call,
    so its rate is not an HBM roofline figure: the per-step line above is.
    Calls are repeated for about half a second after one untimed call."""
    import torch

    import paper_2110_04175_gb300 as rs

    if not run.trees:
        raise RuntimeError("run_fused needs the resident run (run_e2e frees it)")
    K = args.fused_steps
    run.steps(K, w.lr, w.seed, stream)
    torch.cuda.synchronize(dev)
    probe = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    probe[0].record(stream)
    run.steps(K, w.lr, w.seed, stream)
    probe[1].record(stream)
    torch.cuda.synchronize(dev)
    calls = max(1, min(1000, int(500.0 / max(probe[0].elapsed_time(probe[1]), 1e-3))))
    calls = int(reduce_max(float(calls), world))  # the same count on every rank
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    barrier(world)
    torch.cuda.synchronize(dev)
    ev[0].record(stream)
    for _ in range(calls):
        run.steps(K, w.lr, w.seed, stream)
    ev[1].record(stream)
    torch.cuda.synchronize(dev)
    ms = reduce_max(ev[0].elapsed_time(ev[1]), world)
    fused = all(rs.relay_get_steps_kernel(tr.h) == rs.RELAY_KERNEL_FUSED for tr in run.trees)
    E, state_rows = w.E, {"sgd": 0, "nesterov": 1, "adam": 2}[args.optimizer]
    mu_rows = {"stored": w.n, "generated": 0}[run.objective_source]
    # per launch of at most 64 steps: read x, mu, the state, m^{t0-1}; write x, the state and
    # the last two steps' messages
    chunks = -(-K // 64)
    per_call = 0
    for j in range(chunks):
        kc = min(64, K - 64 * j)
        per_call += 4 * w.d * (w.n + mu_rows + state_rows * w.n + E + w.n + state_rows * w.n + min(kc, 2) * E)
    launches = chunks * (1 + (E > 0 or args.algorithm == "dme")) if fused else 2 * K
    return {"value": round(world * K * calls / (ms / 1e3), 4), "unit": "steps/s", "steps_per_call": K,
            "calls": calls, "ms_per_step": round(ms / (K * calls), 5),
            "kernel": "relay_fused_steps_kernel" if fused else "one relay_step per step (a wide node)",
            "launches_per_call": launches * len(run.trees),
            "hbm_bytes_per_call": per_call if fused else None,
            "note": "several steps per launch, the state on chip between them; not an HBM roofline figure"}


def run_graphed(args, w, run, dev, stream, rank: int, world: int):
    """Timed region = one replay of a CUDA graph holding the K steps (for
    launch-bound small problems).  The graph is captured after the warm-up
    and replayed once untimed first (the first launch of a graph also
    uploads it); the timed replay runs the same K steps again."""
    import torch
    torch.cuda.synchronize(dev)
    g = run.capture(args.steps, w.lr, w.seed)
    g.replay()
    torch.cuda.synchronize(dev)
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    barrier(world)
    with ClockSampler(bus_id_of(dev.index or 0) if rank == 0 else None) as clocks:
        start.record(stream)
        g.replay()
        end.record(stream)
        torch.cuda.synchronize(dev)
    total_ms = reduce_max(start.elapsed_time(end), world)
    if rank != 0:
        return
    alg = w.bytes_per_step()
    peak = measured_peaks().get("hbm_gbs") or FALLBACK_HBM_GBS
    per_step = total_ms / args.steps
    line = {"metric": METRIC, "value": round(world * args.steps / (total_ms / 1e3), 2),
            "unit": "steps/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(per_step, 5), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": dict(workload_config(w, world, args), launch="one CUDA graph of K steps"),
            "roofline": {"bound": "hbm", "achieved": round(alg / (per_step / 1e3) / 1e9, 1),
                         "peak": peak, "unit": "GB/s",
                         "frac": round(alg / (per_step / 1e3) / 1e9 / peak, 4), "traffic": None,
                         "kernel": "whole step (graph replay)"},
            "cpu_baseline": None, "e2e": None, "gpu_launches": world * 2 * len(run.trees) * args.steps,
            "clocks": clocks.summary()}
    print(json.dumps(line), flush=True)


def host_mem_available() -> int:
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    return int(line.split()[1]) * 1024
    except OSError:
        pass
    return 0


def pinned_like(t):
    """A page-locked host tensor shaped like `t` (torch's pinned allocator)."""
    import torch
    return torch.empty(t.shape, dtype=t.dtype, pin_memory=True)


def host_link_gbs(dev, mib: int = 1024, reps: int = 4) -> dict:
    """Measured copy rates of this GPU's host link with pinned memory and the
    copy engines: host-to-device alone, device-to-host alone, and both at
    once on two streams (the e2e path's ceiling)."""
    import torch
    n = mib << 18  # floats
    hin = torch.ones(n, dtype=torch.float32, pin_memory=True)
    hout = torch.empty(n, dtype=torch.float32, pin_memory=True)
    din = torch.empty(n, dtype=torch.float32, device=dev)
    dout = torch.zeros(n, dtype=torch.float32, device=dev)
    s1, s2 = torch.cuda.Stream(dev), torch.cuda.Stream(dev)

    def timed(h2d: bool, d2h: bool) -> float:
        torch.cuda.synchronize(dev)
        t0 = time.perf_counter()
        for _ in range(reps):
            if h2d:
                with torch.cuda.stream(s1):
                    din.copy_(hin, non_blocking=True)
            if d2h:
                with torch.cuda.stream(s2):
                    hout.copy_(dout, non_blocking=True)
        torch.cuda.synchronize(dev)
        return (int(h2d) + int(d2h)) * reps * n * 4 / (time.perf_counter() - t0) / 1e9

    timed(True, True)  # warm-up
    out = {"h2d_gbs": timed(True, False), "d2h_gbs": timed(False, True),
           "both_gbs": timed(True, True)}
    del hin, hout, din, dout
    return {k: round(v, 1) for k, v in out.items()}


def run_e2e(args, w, run, dev, stream, world: int):
    """The same metric through the host-state API: x, both message buffers and
    the counters live in pinned host memory, and every step is one
    relay_step_host call that streams them through the GPU (HostRelayRun),
    copies inside the timed region.  The headline copies every row of m^t
    back (the step's whole result, as relay_step writes it); `state_only`
    copies back only the rows a later step reads."""
    import torch

    from paper_2110_04175_gb300.host_stream import HostRelayRun

    if len(run.trees) > 1 or args.optimizer != "sgd" or args.algorithm != "relaysgd":
        return {"value": None, "unit": "steps/s",
                "skipped": "host-state path measured on single-tree SGD workloads"}
    E = max(2 * (w.n - 1), 1)

    def pow2(b):  # the pinned allocator rounds every block up to a power of two
        return 1 << max(0, int(b - 1).bit_length())
    ld = (w.d + 31) // 32 * 32
    need = pow2(w.n * ld * 4) + 2 * pow2(E * ld * 4)
    # every rank on this node pins its own state: split the host's memory
    local_world = max(1, int(os.environ.get("LOCAL_WORLD_SIZE", str(world))))
    avail = host_mem_available()
    # all ranks take the same decision (they enter a barrier below)
    if reduce_min(1.0 if need <= 0.6 * avail / local_world else 0.0, world) < 0.5:
        return {"value": None, "unit": "steps/s",
                "skipped": f"pinned host state of {need / 1e9:.1f} GB per rank exceeds 60% of the "
                           f"{avail / 1e9:.1f} GB available split over {local_world} rank(s)"}
    # free the resident run's buffers first: the host run needs its own
    del run.trees[:]
    run.x = run.mu = None
    torch.cuda.empty_cache()
    link = host_link_gbs(dev)
    cw = 1 << 22
    host = HostRelayRun(w.n, w.d, w.edges, chunk=cw, device=dev, mode=w.mode,
                        c0=shard_offset(int(os.environ.get("RANK", "0")), w.d), full_output=True)
    host.init(w.x0_std, w.seed, w.mix, w.mu_scale, w.mu_seed, w.sigma)

    def timed(steps: int):
        host.step(w.lr, w.seed)  # warm-up
        host.sync()
        barrier(world)
        t0 = time.perf_counter()
        for _ in range(steps):
            host.step(w.lr, w.seed)
        host.sync()
        ms = reduce_max((time.perf_counter() - t0) * 1e3, world)
        h2d, d2h = host.bytes_per_step()
        return {"value": round(world * steps / (ms / 1e3), 4), "unit": "steps/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "steps": steps,
                "copy_gbs": round((h2d + d2h) * steps / (ms / 1e3) / 1e9, 1),
                "copy_frac": round((h2d + d2h) * steps / (ms / 1e3) / 1e9 / link["both_gbs"], 3)}

    full = timed(args.e2e_steps)
    host.set_full_output(False)
    state_only = timed(args.e2e_steps)
    state_only["note"] = "only the message rows a later step reads come back (not those arriving at leaves)"
    fused = None
    if args.fused_steps > 0:
        # the same host-state path with relay_steps_host: the state crosses
        # the link once per call of K steps (one relay_steps call per chunk)
        K = args.fused_steps
        host.steps(2, w.lr, w.seed)
        host.sync()
        barrier(world)
        t1 = time.perf_counter()
        host.steps(K, w.lr, w.seed)
        host.sync()
        fms = reduce_max((time.perf_counter() - t1) * 1e3, world)
        h2d, d2h = host.bytes_per_step()
        fused = {"value": round(world * K / (fms / 1e3), 4), "unit": "steps/s", "steps_per_call": K,
                 "h2d_bytes_per_call": h2d, "d2h_bytes_per_call": d2h,
                 "note": "relay_steps_host: one relay_steps call per chunk visit"}
    return {**full,
            "path": "relay_step_host (C ABI): state in pinned host memory in the device layout, streamed "
                    f"through the GPU in {host.nchunks} chunks of {cw} coordinates (copy-in / kernel / "
                    "copy-out streams of the library's plan), copies inside the timed region; x and the "
                    "counters both ways, the message rows the step reads in, every row of m^t out",
            "host_link": link, "state_only": state_only, "fused_steps": fused}


def traffic_per_launch(w, objective: str, kernel: str = "relay_models_kernel", optimizer: str = "sgd"):
    """DRAM bytes per launch of the step kernel from the committed ncu
    summary for this kernel, workload, objective source and local optimiser
    (profiles/traffic.txt; plain entries are SGD), or None when no capture of
    the current kernel exists for it."""
    key = f"{kernel}/{w.name}/{objective}" + ("" if optimizer == "sgd" else f"/{optimizer}")
    path = os.path.join(ROOT, "profiles", "traffic.txt")
    try:
        with open(path) as f:
            for line in f:
                parts = line.split()
                if len(parts) == 2 and not line.startswith("#") and parts[0] == key:
                    return int(parts[1])
    except OSError:
        pass
    return None


def main(argv=None):
    p = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawTextHelpFormatter)
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=50)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["native", "reference"], default="native")
    p.add_argument("--workload", default=DEFAULT_WORKLOAD)
    p.add_argument("--e2e-steps", type=int, default=5)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--kernel", choices=["auto", "walk", "nodes"], default="auto",
                   help="step kernel (relay_set_kernel)")
    p.add_argument("--l2-flush", choices=["auto", "on", "off"], default="auto",
                   help="flush L2 before every timed step (auto: when a step's working set is "
                        "under twice the L2)")
    p.add_argument("--optimizer", choices=["sgd", "nesterov", "adam"], default="sgd",
                   help="local optimiser of the local step (appendix: momentum / Adam)")
    p.add_argument("--algorithm", choices=["relaysgd", "grad", "dme"], default="relaysgd",
                   help="Algorithm 1 (default), 6 (relayed updates) or 5 (mean estimation)")
    p.add_argument("--graph", action="store_true",
                   help="time one CUDA-graph replay of the K steps (small, launch-bound workloads)")
    p.add_argument("--lost-prob", type=float, default=0.0,
                   help="probability that each message is lost in transit, per step")
    p.add_argument("--objective", choices=["generated", "stored"], default="stored",
                   help="regenerate the centres mu in the kernel, or read a stored mu array")
    p.add_argument("--fused-steps", type=int, default=64,
                   help="also time relay_steps with this many steps per call (0: skip); reported "
                        "under 'fused_steps', beside the per-step headline")
    p.add_argument("--no-per-workload", dest="per_workload", action="store_false",
                   help="skip the other HBM-bound workloads (reported under 'per_workload')")
    p.add_argument("--d", type=int, default=None,
                   help="override the workload's d (small cases for profiling; not a bench line)")
    args = p.parse_args(argv)
    if args.warmup < 3:
        p.error("--warmup must be >= 3")

    from paper_2110_04175_gb300 import workloads as wl
    w = wl.by_name(args.workload)
    if args.d is not None:
        w.d = args.d
        w.name = f"{w.name}@d={args.d}"
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        run_reference(args, w, rank)
        return
    if world > 1:
        import torch
        import torch.distributed as dist
        n_dev = torch.cuda.device_count()
        torch.cuda.set_device(local_device(int(os.environ.get("LOCAL_RANK", "0")), n_dev))
        local_world = int(os.environ.get("LOCAL_WORLD_SIZE", str(world)))
        dist.init_process_group(process_group_backend(local_world, n_dev))
    try:
        run_native(args, w, rank, world)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
