"""ctypes marshalling for librelaysum.so (see include/relaysum.h)."""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np

from . import build as _build

RELAY_OK = 0
RELAY_EINVAL = -1
RELAY_ENOTTREE = -2
RELAY_ECUDA = -3
RELAY_ENOMEM = -4
RELAY_EUNSUPPORTED = -5
RELAY_MAX_N = 256
RELAY_OPT_SGD = 0
RELAY_OPT_NESTEROV = 1
RELAY_OPT_ADAM = 2
RELAY_ALGO_RELAYSGD = 0
RELAY_ALGO_GRAD = 1
RELAY_ALGO_DME = 2
RELAY_KERNEL_AUTO = 0
RELAY_KERNEL_WALK = 1
RELAY_KERNEL_NODES = 2
RELAY_KERNEL_FUSED = 3
RELAY_HOST_FULL_OUTPUT = 1

_lock = threading.Lock()
_lib = None


def library_path() -> str:
    return _build.LIB


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(_build.LIB):
            raise RuntimeError(
                f"{_build.LIB} is missing: build the CUDA library first "
                "(python -c 'import __graft_entry__ as g; g.build()')")
        lib = ctypes.CDLL(_build.LIB)
        vp, i32, i64, u64, f32 = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64,
                                  ctypes.c_float)
        sig = {
            "relay_create": (ctypes.c_int, [ctypes.POINTER(vp), i32, i64, vp, i32]),
            "relay_destroy": (None, [vp]),
            "relay_ld": (i64, [vp]),
            "relay_num_edges": (i32, [vp]),
            "relay_edges": (ctypes.c_int, [vp, vp, vp]),
            "relay_set_rebuild_mode": (ctypes.c_int, [vp, i32]),
            "relay_set_kernel": (ctypes.c_int, [vp, i32]),
            "relay_set_received_sums": (ctypes.c_int, [vp, i32]),
            "relay_message_rows": (i32, [vp]),
            "relay_get_kernel": (ctypes.c_int, [vp]),
            "relay_get_steps_kernel": (ctypes.c_int, [vp]),
            "relay_set_strides": (ctypes.c_int, [vp, i64, i64]),
            "relay_set_local_optimizer": (ctypes.c_int, [vp, i32, f32, f32, f32, vp, vp]),
            "relay_set_lost_messages": (ctypes.c_int, [vp, vp]),
            "relay_set_algorithm": (ctypes.c_int, [vp, i32, vp]),
            "relay_set_coord_offset": (ctypes.c_int, [vp, i64]),
            "relay_set_objective": (ctypes.c_int, [vp, vp, f32]),
            "relay_set_objective_generated": (ctypes.c_int, [vp, vp, i32, f32, u64, f32]),
            "relay_fill_objective": (ctypes.c_int, [vp, vp, vp, i32, f32, u64, vp]),
            "relay_init": (ctypes.c_int, [vp, vp, vp, vp, vp, f32, u64, vp]),
            "relay_step_counts": (ctypes.c_int, [vp, vp, vp]),
            "relay_step_models": (ctypes.c_int, [vp, vp, vp, vp, vp, f32, u64, i64, vp]),
            "relay_step": (ctypes.c_int, [vp, vp, vp, vp, vp, f32, u64, i64, vp]),
            "relay_steps": (ctypes.c_int, [vp, vp, vp, vp, vp, f32, u64, i64, i64, vp]),
            "relay_step_windows": (ctypes.c_int, [vp, i32, vp, vp, vp, vp, f32, u64, i64, vp]),
            "relay_host_staging_bytes": (i64, [vp, i64, i32]),
            "relay_host_plan_create": (ctypes.c_int, [ctypes.POINTER(vp), vp, i64, i32, vp, i64, i32]),
            "relay_host_plan_destroy": (None, [vp]),
            "relay_host_bytes": (ctypes.c_int, [vp, vp, vp]),
            "relay_step_host": (ctypes.c_int, [vp, vp, vp, vp, vp, f32, u64, i64, vp]),
            "relay_steps_host": (ctypes.c_int, [vp, vp, vp, vp, vp, f32, u64, i64, i64, vp]),
            "relay_nbar": (ctypes.c_int, [vp, vp, vp]),
            "relay_program": (ctypes.c_int, [vp, vp, vp, vp, vp]),
            "relay_metrics_workspace": (i64, [vp]),
            "relay_metrics": (ctypes.c_int, [vp, vp, vp, vp, vp]),
            "relay_metrics_static": (ctypes.c_int, [vp, vp, vp, vp]),
            "relay_error_string": (ctypes.c_char_p, [ctypes.c_int]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


class RelayError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {relay_error_string(status)} ({status})")


def relay_error_string(status: int) -> str:
    return _load().relay_error_string(int(status)).decode()


def _check(status: int, what: str):
    if status != RELAY_OK:
        raise RelayError(status, what)


def _ptr(t) -> int | None:
    """Device or host address of a torch tensor / numpy array / int; None for NULL."""
    if t is None:
        return None
    if isinstance(t, int):
        return t or None
    if isinstance(t, np.ndarray):
        return t.ctypes.data or None
    return t.data_ptr() or None


def _stream(stream) -> int | None:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream or None
    if isinstance(stream, int):
        return stream or None
    return stream.cuda_stream or None


class RelayHandle:
    """Owns a relay_handle*; destroyed with the object or by relay_destroy."""

    def __init__(self, raw: int, n: int, d: int):
        self.raw = raw
        self.n = n
        self.d = d
        self._lib = _load()

    def __del__(self):
        if getattr(self, "raw", None):
            self._lib.relay_destroy(self.raw)
            self.raw = None

    @property
    def ld(self) -> int:
        return relay_ld(self)

    @property
    def E(self) -> int:
        return relay_num_edges(self)


def _h(h) -> int:
    return h.raw if isinstance(h, RelayHandle) else int(h)


def relay_create(n: int, d: int, edges) -> RelayHandle:
    lib = _load()
    e = np.ascontiguousarray(np.asarray(edges, dtype=np.int32).reshape(-1, 2))
    out = ctypes.c_void_p()
    _check(lib.relay_create(ctypes.byref(out), int(n), int(d), e.ctypes.data if e.size else None,
                            int(e.shape[0])), "relay_create")
    return RelayHandle(out.value, int(n), int(d))


def relay_destroy(h: RelayHandle):
    if isinstance(h, RelayHandle):
        if h.raw:
            _load().relay_destroy(h.raw)
            h.raw = None
    else:
        _load().relay_destroy(int(h))


def relay_ld(h) -> int:
    return int(_load().relay_ld(_h(h)))


def relay_num_edges(h) -> int:
    return int(_load().relay_num_edges(_h(h)))


def relay_edges(h):
    E = relay_num_edges(h)
    src = np.zeros(max(E, 1), dtype=np.int32)
    dst = np.zeros(max(E, 1), dtype=np.int32)
    _check(_load().relay_edges(_h(h), src.ctypes.data, dst.ctypes.data), "relay_edges")
    return src[:E], dst[:E]


def relay_set_rebuild_mode(h, mode: int):
    _check(_load().relay_set_rebuild_mode(_h(h), int(mode)), "relay_set_rebuild_mode")


def relay_set_kernel(h, kernel: int):
    _check(_load().relay_set_kernel(_h(h), int(kernel)), "relay_set_kernel")


def relay_set_received_sums(h, enable: bool):
    _check(_load().relay_set_received_sums(_h(h), int(bool(enable))), "relay_set_received_sums")


def relay_message_rows(h) -> int:
    r = int(_load().relay_message_rows(_h(h)))
    _check(min(r, 0), "relay_message_rows")
    return r


def relay_get_kernel(h) -> int:
    k = _load().relay_get_kernel(_h(h))
    _check(min(k, 0), "relay_get_kernel")
    return k


def relay_get_steps_kernel(h) -> int:
    """RELAY_KERNEL_FUSED when relay_steps runs several steps per launch, else
    the per-step kernel it repeats."""
    k = _load().relay_get_steps_kernel(_h(h))
    _check(min(k, 0), "relay_get_steps_kernel")
    return k


def relay_set_strides(h, ld_x: int, ld_msg: int):
    _check(_load().relay_set_strides(_h(h), int(ld_x), int(ld_msg)), "relay_set_strides")


def relay_set_local_optimizer(h, kind: int, beta1: float = 0.0, beta2: float = 0.0,
                              eps: float = 0.0, state1=None, state2=None):
    _check(_load().relay_set_local_optimizer(_h(h), int(kind), float(beta1), float(beta2),
                                             float(eps), _ptr(state1), _ptr(state2)),
           "relay_set_local_optimizer")


def relay_set_algorithm(h, algo: int, dme_count=None):
    _check(_load().relay_set_algorithm(_h(h), int(algo), _ptr(dme_count)), "relay_set_algorithm")


def relay_set_lost_messages(h, lost=None):
    """lost: host array of E flags (non-zero = lost) or None."""
    if lost is None:
        _check(_load().relay_set_lost_messages(_h(h), None), "relay_set_lost_messages")
        return
    m = np.ascontiguousarray(np.asarray(lost, dtype=np.uint8))
    _check(_load().relay_set_lost_messages(_h(h), m.ctypes.data if m.size else None),
           "relay_set_lost_messages")


def relay_set_coord_offset(h, c0: int):
    _check(_load().relay_set_coord_offset(_h(h), int(c0)), "relay_set_coord_offset")


def relay_set_objective(h, mu, sigma: float):
    _check(_load().relay_set_objective(_h(h), _ptr(mu), float(sigma)), "relay_set_objective")


def relay_set_objective_generated(h, mix, K: int, mu_scale: float, mu_seed: int, sigma: float):
    """mix: host float32 [n][K] (numpy); the kernel regenerates mu from it."""
    m = np.ascontiguousarray(np.asarray(mix, dtype=np.float32))
    _check(_load().relay_set_objective_generated(_h(h), m.ctypes.data if m.size else None, int(K),
                                                 float(mu_scale), int(mu_seed), float(sigma)),
           "relay_set_objective_generated")


def relay_fill_objective(h, mu, mix, K: int, mu_scale: float, mu_seed: int, stream=None):
    _check(_load().relay_fill_objective(_h(h), _ptr(mu), _ptr(mix), int(K), float(mu_scale),
                                        int(mu_seed), _stream(stream)), "relay_fill_objective")


def relay_init(h, x, msg_a, msg_b, counts, x0_std: float, seed: int, stream=None):
    _check(_load().relay_init(_h(h), _ptr(x), _ptr(msg_a), _ptr(msg_b), _ptr(counts),
                              float(x0_std), int(seed), _stream(stream)), "relay_init")


def relay_step_counts(h, counts, stream=None):
    _check(_load().relay_step_counts(_h(h), _ptr(counts), _stream(stream)), "relay_step_counts")


def relay_step_models(h, x, msg_in, msg_out, counts, lr: float, seed: int, step: int, stream=None):
    _check(_load().relay_step_models(_h(h), _ptr(x), _ptr(msg_in), _ptr(msg_out), _ptr(counts),
                                     float(lr), int(seed), int(step), _stream(stream)),
           "relay_step_models")


def relay_step(h, x, msg_in, msg_out, counts, lr: float, seed: int, step: int, stream=None):
    _check(_load().relay_step(_h(h), _ptr(x), _ptr(msg_in), _ptr(msg_out), _ptr(counts),
                              float(lr), int(seed), int(step), _stream(stream)), "relay_step")


def relay_step_windows(hs, xs, msg_ins, msg_outs, counts, lr: float, seed: int, step: int, stream=None):
    """relay_step over the tree windows hs[k] (x, messages, counters per window),
    in one launch of the step kernel where the windows allow it."""
    k = len(hs)
    arr = ctypes.c_void_p * max(k, 1)
    _check(_load().relay_step_windows(arr(*[_h(h) for h in hs]), k, arr(*[_ptr(v) for v in xs]),
                                      arr(*[_ptr(v) for v in msg_ins]), arr(*[_ptr(v) for v in msg_outs]),
                                      arr(*[_ptr(v) for v in counts]), float(lr), int(seed), int(step),
                                      _stream(stream)), "relay_step_windows")


class RelayHostPlan:
    """Owns a relay_host_plan* (and keeps its handle and staging alive)."""

    def __init__(self, raw: int, h, staging):
        self.raw, self.h, self.staging = raw, h, staging
        self._lib = _load()

    def __del__(self):
        if getattr(self, "raw", None):
            self._lib.relay_host_plan_destroy(self.raw)
            self.raw = None


def relay_host_staging_bytes(h, chunk: int, buffers: int) -> int:
    r = int(_load().relay_host_staging_bytes(_h(h), int(chunk), int(buffers)))
    _check(min(r, 0), "relay_host_staging_bytes")
    return r


def relay_host_plan_create(h, chunk: int, buffers: int, staging, flags: int = 0) -> RelayHostPlan:
    """staging: a device tensor of at least relay_host_staging_bytes bytes."""
    out = ctypes.c_void_p()
    _check(_load().relay_host_plan_create(ctypes.byref(out), _h(h), int(chunk), int(buffers), _ptr(staging),
                                          int(staging.numel() * staging.element_size()), int(flags)),
           "relay_host_plan_create")
    return RelayHostPlan(out.value, h, staging)


def relay_host_bytes(plan) -> tuple:
    h2d, d2h = ctypes.c_int64(), ctypes.c_int64()
    _check(_load().relay_host_bytes(plan.raw, ctypes.addressof(h2d), ctypes.addressof(d2h)), "relay_host_bytes")
    return int(h2d.value), int(d2h.value)


def relay_step_host(plan, x, msg_in, msg_out, counts, lr: float, seed: int, step: int, stream=None):
    _check(_load().relay_step_host(plan.raw, _ptr(x), _ptr(msg_in), _ptr(msg_out), _ptr(counts), float(lr),
                                   int(seed), int(step), _stream(stream)), "relay_step_host")


def relay_steps_host(plan, x, msg_in, msg_out, counts, lr: float, seed: int, t0: int, k: int, stream=None):
    _check(_load().relay_steps_host(plan.raw, _ptr(x), _ptr(msg_in), _ptr(msg_out), _ptr(counts), float(lr),
                                    int(seed), int(t0), int(k), _stream(stream)), "relay_steps_host")


def relay_steps(h, x, msg_a, msg_b, counts, lr: float, seed: int, t0: int, k: int, stream=None):
    """k steps t0 .. t0+k-1 in one launch per 64 steps; msg_a holds m^{t0-1}, and the
    result equals k relay_step calls alternating msg_a and msg_b, bit for bit."""
    _check(_load().relay_steps(_h(h), _ptr(x), _ptr(msg_a), _ptr(msg_b), _ptr(counts),
                               float(lr), int(seed), int(t0), int(k), _stream(stream)), "relay_steps")


def relay_metrics_workspace(h) -> int:
    return int(_load().relay_metrics_workspace(_h(h)))


def relay_metrics(h, x, workspace, out, stream=None):
    """out (device float64 [2]) = (consensus distance, distance to the optimum)."""
    _check(_load().relay_metrics(_h(h), _ptr(x), _ptr(workspace), _ptr(out), _stream(stream)),
           "relay_metrics")


def relay_metrics_static(h, x, out, stream=None):
    """relay_metrics with the library's built-in scratch: allocates nothing."""
    _check(_load().relay_metrics_static(_h(h), _ptr(x), _ptr(out), _stream(stream)),
           "relay_metrics_static")


def relay_nbar(h, counts_host) -> np.ndarray:
    c = np.ascontiguousarray(np.asarray(counts_host, dtype=np.int32))
    n = h.n if isinstance(h, RelayHandle) else None
    if n is None:
        raise ValueError("relay_nbar needs a RelayHandle")
    out = np.zeros(n, dtype=np.int32)
    _check(_load().relay_nbar(_h(h), c.ctypes.data if c.size else None, out.ctypes.data),
           "relay_nbar")
    return out


def relay_program(h):
    """(nslots, order[n], node_rec[n][12], pos_rec[E][4]) of the step kernels' visit program."""
    n, E = h.n, relay_num_edges(h)
    nslots = ctypes.c_int32()
    order = np.zeros(n, dtype=np.int32)
    node = np.zeros((n, 12), dtype=np.int32)
    pos = np.zeros((max(E, 1), 4), dtype=np.int32)
    _check(_load().relay_program(_h(h), ctypes.addressof(nslots), order.ctypes.data,
                                 node.ctypes.data, pos.ctypes.data), "relay_program")
    return int(nslots.value), order, node, pos[:E]


class _TreeState:
    """One tree of a run: its handle, column window, messages and counters."""

    def __init__(self, h, col0: int, d: int, E: int, msg, counts):
        self.h, self.col0, self.d, self.E = h, col0, d, E
        self.msg = msg          # two [rows][ld_msg] buffers (double buffering): E messages, then
                                # the received sums of the wide nodes, if any
        self.counts = counts    # int32 [E]
        self.cur = 0            # msg[cur] holds m^{t-1}

    @property
    def messages(self):
        return self.msg[self.cur]


def _window_ptr(t, col0: int) -> int:
    return t.data_ptr() + 4 * col0


class RelayRun:
    """Device state of one RelaySGD run, allocated with torch on `device`.

    `edges` is one tree, or a list of trees that split the coordinates into
    contiguous quad-aligned windows of the same model array -- the double
    binary trees of Section 3 are a list of two.  Buffers: x [n][ld], per tree
    two message buffers [rows][ld_tree] (double buffering; rows = E plus the
    wide nodes' received sums) and counters int32 [E], and -- for
    objective="stored" -- the centres mu [n][ld] (objective="generated" lets
    the kernel regenerate them).  ``step()`` enqueues one step on the current
    torch stream: relay_step, or relay_step_windows for several trees.
    """

    def __init__(self, n: int, d: int, edges, device="cuda", mode: int = 1, c0: int = 0,
                 objective: str = "stored", optimizer=None, algorithm: str = "relaysgd",
                 kernel: str = "auto", received_sums: bool = True):
        """optimizer: None (SGD), ("nesterov", beta1) or ("adam", beta1, beta2, eps);
        algorithm: "relaysgd" (Alg. 1), "grad" (Alg. 6) or "dme" (Alg. 5, x holds
        the running sums y and `dme_count` the counts s of each tree);
        kernel: "auto", "walk" or "nodes" (relay_set_kernel);
        received_sums: message buffers carry the wide nodes' received sums
        (relay_set_received_sums; no effect on trees without a node of degree > 4)."""
        import torch
        if objective not in ("stored", "generated"):
            raise ValueError(f"objective must be 'stored' or 'generated', not {objective!r}")
        if kernel not in ("auto", "walk", "nodes"):
            raise ValueError(f"kernel must be 'auto', 'walk' or 'nodes', not {kernel!r}")
        trees = list(edges) if isinstance(edges, (list, tuple)) else [edges]
        self.objective = objective
        self.n, self.d, self.c0 = n, d, c0
        self.device = torch.device(device)
        self.ld = (d + 31) // 32 * 32
        f32 = dict(dtype=torch.float32, device=self.device)
        self.x = torch.empty(n, self.ld, **f32)
        self.mu = torch.empty(n, self.ld, **f32) if objective == "stored" else None
        self.objective_source = objective
        kind = {None: RELAY_OPT_SGD, "nesterov": RELAY_OPT_NESTEROV, "adam": RELAY_OPT_ADAM}[
            optimizer[0] if optimizer else None]
        self.state = [torch.empty(n, self.ld, **f32) for _ in range(kind)]  # m (and v)
        nq = (d + 3) // 4
        self.trees = []
        for k, tree_edges in enumerate(trees):
            q_lo, q_hi = nq * k // len(trees), nq * (k + 1) // len(trees)
            col0 = 4 * q_lo
            dk = min(4 * q_hi, d) - col0 if q_hi > q_lo else 0
            h = relay_create(n, dk, tree_edges)
            relay_set_received_sums(h, received_sums)
            relay_set_rebuild_mode(h, mode)
            relay_set_kernel(h, {"auto": RELAY_KERNEL_AUTO, "walk": RELAY_KERNEL_WALK,
                                 "nodes": RELAY_KERNEL_NODES}[kernel])
            relay_set_coord_offset(h, c0 + col0)
            ld_m = relay_ld(h)
            relay_set_strides(h, self.ld, ld_m)
            if kind != RELAY_OPT_SGD:
                hyper = list(optimizer[1:]) + [0.0] * (3 - len(optimizer[1:]))
                st = [_window_ptr(t, col0) if dk > 0 else None for t in self.state] + [None]
                relay_set_local_optimizer(h, kind, hyper[0], hyper[1], hyper[2], st[0], st[1])
            algo = {"relaysgd": RELAY_ALGO_RELAYSGD, "grad": RELAY_ALGO_GRAD,
                    "dme": RELAY_ALGO_DME}[algorithm]
            dme_count = (torch.zeros(n, dtype=torch.int64, device=self.device)
                         if algo == RELAY_ALGO_DME else None)
            relay_set_algorithm(h, algo, dme_count)
            E = relay_num_edges(h)
            rows = relay_message_rows(h)  # E, + the wide nodes' received sums
            msg = [torch.empty(max(rows, 1), max(ld_m, 1), **f32) for _ in range(2)]
            counts = torch.zeros(max(E, 1), dtype=torch.int32, device=self.device)
            tr = _TreeState(h, col0, dk, E, msg, counts)
            tr.dme_count = dme_count
            self.trees.append(tr)
        self.t = 0

    # single-tree conveniences
    @property
    def h(self):
        return self.trees[0].h

    @property
    def E(self) -> int:
        return self.trees[0].E

    @property
    def counts(self):
        return self.trees[0].counts

    @property
    def msg(self):
        return self.trees[0].msg

    @property
    def cur(self) -> int:
        return self.trees[0].cur

    @cur.setter
    def cur(self, v: int):
        self.trees[0].cur = v

    @property
    def messages(self):
        """m^{t-1} of the first tree: the messages of the last step."""
        return self.trees[0].messages

    def _x(self, tr):
        return _window_ptr(self.x, tr.col0) if tr.d > 0 else None

    def init(self, x0_std: float, seed: int, mix, mu_scale: float, mu_seed: int, sigma: float):
        import torch
        mix = np.asarray(mix, dtype=np.float32)
        mix_t = None
        for tr in self.trees:
            if self.objective == "stored":
                if mix_t is None:
                    mix_t = torch.as_tensor(mix, device=self.device).contiguous()
                mu = _window_ptr(self.mu, tr.col0) if tr.d > 0 else None
                relay_fill_objective(tr.h, mu, mix_t, mix_t.shape[1], mu_scale, mu_seed)
                relay_set_objective(tr.h, mu, sigma)
            else:
                relay_set_objective_generated(tr.h, mix, mix.shape[1], mu_scale, mu_seed, sigma)
            relay_init(tr.h, self._x(tr), tr.msg[0], tr.msg[1], tr.counts, x0_std, seed)
            tr.cur = 0
        self._mix = mix_t  # keep alive until the fills have run
        self.t = 0

    def metrics(self):
        """(consensus distance, distance of the average model to the optimum)
        of the current models, as a device float64 tensor [trees][2]."""
        import torch
        out = torch.zeros(len(self.trees), 2, dtype=torch.float64, device=self.device)
        for k, tr in enumerate(self.trees):
            if tr.d == 0:
                continue
            ws = torch.empty(relay_metrics_workspace(tr.h), dtype=torch.float64, device=self.device)
            relay_metrics(tr.h, self._x(tr), ws, out[k])
        return out

    def state_dict(self) -> dict:
        """The run's full state as host tensors: models, both message buffers,
        counters, optimiser state, mean-estimation counts, step and buffer
        parity.  With the seeds, it resumes the run bit for bit."""
        sd = {"t": self.t, "x": self.x.cpu(), "state": [s.cpu() for s in self.state],
              "trees": [{"cur": tr.cur, "msg": [m.cpu() for m in tr.msg],
                         "counts": tr.counts.cpu(),
                         "dme_count": None if tr.dme_count is None else tr.dme_count.cpu()}
                        for tr in self.trees]}
        return sd

    def load_state_dict(self, sd: dict):
        """Restores a state_dict() into this run (same n, d, trees and options;
        init() must have bound the objective first)."""
        self.t = int(sd["t"])
        self.x.copy_(sd["x"])
        for dst, src in zip(self.state, sd["state"]):
            dst.copy_(src)
        for tr, st in zip(self.trees, sd["trees"]):
            tr.cur = int(st["cur"])
            for dst, src in zip(tr.msg, st["msg"]):
                dst.copy_(src)
            tr.counts.copy_(st["counts"])
            if tr.dme_count is not None:
                tr.dme_count.copy_(st["dme_count"])

    def capture(self, steps: int, lr: float, seed: int):
        """Records the next `steps` steps (t, t+1, ...) into one CUDA graph and
        advances the run's bookkeeping as if they had run: replay the returned
        graph exactly once to run them (the step counters are fixed in it).
        For launch-bound small problems this replaces 2 launches per tree and
        step by one graph launch."""
        import torch
        g = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream(self.device)
        side.wait_stream(torch.cuda.current_stream(self.device))
        with torch.cuda.graph(g, stream=side):
            for _ in range(steps):
                self.step(lr, seed, side)
        return g

    def set_lost(self, lost, tree: int = 0):
        """Messages of the next steps lost in transit on tree `tree` (E flags or None)."""
        relay_set_lost_messages(self.trees[tree].h, lost)

    def _per_tree(self, issue, stream):
        """Calls issue(tree, stream) for every tree.  One tree
        runs on `stream` (default: the current stream).  With several trees
        (double binary trees) the windows, which share no data, run on
        streams forked from `stream` and joined back to it, so one window's
        last wave overlaps the next window's start."""
        if len(self.trees) == 1:
            issue(self.trees[0], stream)
            return
        import torch
        if stream is None:
            main = torch.cuda.current_stream(self.device)
        elif isinstance(stream, int):
            main = torch.cuda.ExternalStream(stream) if stream else torch.cuda.default_stream(self.device)
        else:
            main = stream
        if getattr(self, "_side", None) is None:
            self._side = [torch.cuda.Stream(self.device) for _ in self.trees]
        fork = torch.cuda.Event()
        fork.record(main)
        joins = []
        for tr, side in zip(self.trees, self._side):
            side.wait_event(fork)
            issue(tr, side)
            done = torch.cuda.Event()
            done.record(side)
            joins.append(done)
        for done in joins:
            main.wait_event(done)

    def step(self, lr: float, seed: int, stream=None):
        """Enqueues one step on `stream` (default: the current stream): relay_step,
        or with several tree windows one relay_step_windows call (one counter
        launch and one step-kernel launch for the windows where they allow it;
        it measured the same as the windows on forked streams, step_forked)."""
        trs = self.trees
        if len(trs) == 1:
            tr = trs[0]
            relay_step(tr.h, self._x(tr), tr.msg[tr.cur], tr.msg[1 - tr.cur], tr.counts, lr, seed, self.t, stream)
        else:
            relay_step_windows([tr.h for tr in trs], [self._x(tr) for tr in trs], [tr.msg[tr.cur] for tr in trs],
                               [tr.msg[1 - tr.cur] for tr in trs], [tr.counts for tr in trs], lr, seed, self.t,
                               stream)
        for tr in trs:
            tr.cur = 1 - tr.cur
        self.t += 1

    def step_forked(self, lr: float, seed: int, stream=None):
        """The same step with one relay_step per tree window, the windows on
        streams forked from `stream` and joined back (the same bits as step())."""
        def issue(tr, s):
            relay_step(tr.h, self._x(tr), tr.msg[tr.cur], tr.msg[1 - tr.cur], tr.counts, lr, seed, self.t, s)
            tr.cur = 1 - tr.cur

        self._per_tree(issue, stream)
        self.t += 1

    def steps(self, k: int, lr: float, seed: int, stream=None):
        """Enqueues k steps with relay_steps (the models and messages stay on
        chip between them): the same state, bit for bit, as k step() calls."""
        k = int(k)

        def issue(tr, s):
            relay_steps(tr.h, self._x(tr), tr.msg[tr.cur], tr.msg[1 - tr.cur], tr.counts, lr, seed, self.t, k, s)
            tr.cur ^= k & 1

        self._per_tree(issue, stream)
        self.t += k
