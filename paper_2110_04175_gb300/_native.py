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
            "relay_set_coord_offset": (ctypes.c_int, [vp, i64]),
            "relay_set_objective": (ctypes.c_int, [vp, vp, f32]),
            "relay_fill_objective": (ctypes.c_int, [vp, vp, vp, i32, f32, u64, vp]),
            "relay_init": (ctypes.c_int, [vp, vp, vp, vp, vp, f32, u64, vp]),
            "relay_step_counts": (ctypes.c_int, [vp, vp, vp]),
            "relay_step_models": (ctypes.c_int, [vp, vp, vp, vp, vp, f32, u64, i64, vp]),
            "relay_step": (ctypes.c_int, [vp, vp, vp, vp, vp, f32, u64, i64, vp]),
            "relay_nbar": (ctypes.c_int, [vp, vp, vp]),
            "relay_program": (ctypes.c_int, [vp, vp, vp, vp, vp]),
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


def relay_set_coord_offset(h, c0: int):
    _check(_load().relay_set_coord_offset(_h(h), int(c0)), "relay_set_coord_offset")


def relay_set_objective(h, mu, sigma: float):
    _check(_load().relay_set_objective(_h(h), _ptr(mu), float(sigma)), "relay_set_objective")


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
    """(nslots, order[n], node_rec[n][8], pos_rec[E][3]) of the fused kernel's visit program."""
    n, E = h.n, relay_num_edges(h)
    nslots = ctypes.c_int32()
    order = np.zeros(n, dtype=np.int32)
    node = np.zeros((n, 8), dtype=np.int32)
    pos = np.zeros((max(E, 1), 3), dtype=np.int32)
    _check(_load().relay_program(_h(h), ctypes.addressof(nslots), order.ctypes.data,
                                 node.ctypes.data, pos.ctypes.data), "relay_program")
    return int(nslots.value), order, node, pos[:E]


class RelayRun:
    """Device state of one RelaySGD run, allocated with torch on `device`.

    Buffers: x [n][ld], mu [n][ld], two message buffers [E][ld] (double
    buffering), counts int32 [E].  ``step()`` enqueues one relay_step on the
    current torch stream and swaps the message buffers.
    """

    def __init__(self, n: int, d: int, edges, device="cuda", mode: int = 1, c0: int = 0):
        import torch
        self.h = relay_create(n, d, edges)
        relay_set_rebuild_mode(self.h, mode)
        relay_set_coord_offset(self.h, c0)
        self.n, self.d, self.E, self.ld = n, d, relay_num_edges(self.h), relay_ld(self.h)
        self.device = torch.device(device)
        f32 = dict(dtype=torch.float32, device=self.device)
        self.x = torch.empty(n, self.ld, **f32)
        self.mu = torch.empty(n, self.ld, **f32)
        self.msg = [torch.empty(max(self.E, 1), self.ld, **f32) for _ in range(2)]
        self.counts = torch.zeros(max(self.E, 1), dtype=torch.int32, device=self.device)
        self.t = 0
        self.cur = 0  # msg[cur] holds m^{t-1}

    def init(self, x0_std: float, seed: int, mix, mu_scale: float, mu_seed: int, sigma: float):
        import torch
        mix_t = torch.as_tensor(np.asarray(mix, dtype=np.float32), device=self.device).contiguous()
        relay_fill_objective(self.h, self.mu, mix_t, mix_t.shape[1], mu_scale, mu_seed)
        relay_set_objective(self.h, self.mu, sigma)
        relay_init(self.h, self.x, self.msg[0], self.msg[1], self.counts, x0_std, seed)
        self._mix = mix_t  # keep alive until the fill has run
        self.t = 0
        self.cur = 0

    def step(self, lr: float, seed: int, stream=None):
        relay_step(self.h, self.x, self.msg[self.cur], self.msg[1 - self.cur], self.counts, lr,
                   seed, self.t, stream)
        self.cur = 1 - self.cur
        self.t += 1

    @property
    def messages(self):
        """m^{t-1}: the messages of the last step."""
        return self.msg[self.cur]
