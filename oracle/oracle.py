"""ctypes wrapper around the plain-C RelaySum oracle (relaysum_oracle.c).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may use this module; the product path
(``paper_2110_04175_gb300``) never imports it, and this module imports nothing
from the product package.

All floating-point arrays are numpy float64, row-major ``[rows][len]``.
What is computed is Algorithm 1 (RelaySGD) of Vogels et al., arXiv 2110.04175,
with the robust rebuild of its Section 4.4 as mode 1; the C file's header
states the equations.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "relaysum_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

ORACLE_OK = 0
ORACLE_EINVAL = -1
ORACLE_ENOTTREE = -2
ORACLE_ENOMEM = -3


def build(force: bool = False) -> str:
    """Compiles the oracle with gcc (no FMA contraction, no fast-math)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.run(
            ["gcc", "-O2", "-std=c11", "-Wall", "-Wextra", "-ffp-contract=off",
             "-fno-fast-math", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"],
            check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        i32p = ctypes.POINTER(ctypes.c_int32)
        u32p = ctypes.POINTER(ctypes.c_uint32)
        f64p = ctypes.POINTER(ctypes.c_double)
        lib.oracle_philox4x32_10.argtypes = [u32p, u32p, u32p]
        lib.oracle_philox4x32_10.restype = None
        lib.oracle_uniform.argtypes = [ctypes.c_uint32]
        lib.oracle_uniform.restype = ctypes.c_double
        lib.oracle_normal.argtypes = [ctypes.c_uint64, ctypes.c_int64, ctypes.c_uint32,
                                      ctypes.c_uint32, ctypes.c_uint32]
        lib.oracle_normal.restype = ctypes.c_double
        lib.oracle_fill_normals.argtypes = [ctypes.c_uint64, ctypes.c_int64, ctypes.c_int64,
                                            ctypes.c_uint32, ctypes.c_uint32, ctypes.c_uint32, f64p]
        lib.oracle_fill_normals.restype = ctypes.c_int
        lib.oracle_fill_mu.argtypes = [ctypes.c_int, ctypes.c_int, f64p, ctypes.c_double,
                                       ctypes.c_uint64, ctypes.c_int64, ctypes.c_int64, f64p]
        lib.oracle_fill_mu.restype = ctypes.c_int
        lib.oracle_fill_x0.argtypes = [ctypes.c_int, ctypes.c_double, ctypes.c_uint64,
                                       ctypes.c_int64, ctypes.c_int64, f64p]
        lib.oracle_fill_x0.restype = ctypes.c_int
        lib.oracle_run.argtypes = [ctypes.c_int, i32p, ctypes.c_int, ctypes.c_int64,
                                   ctypes.c_int64, f64p, f64p, f64p, i32p, ctypes.c_double,
                                   ctypes.c_double, ctypes.c_uint64, ctypes.c_int64,
                                   ctypes.c_int64, ctypes.c_int, i32p]
        lib.oracle_run.restype = ctypes.c_int
        lib.oracle_run_ext.argtypes = [ctypes.c_int, i32p, ctypes.c_int, ctypes.c_int64,
                                       ctypes.c_int64, f64p, f64p, f64p, i32p, f64p, f64p,
                                       ctypes.c_double, ctypes.c_double, ctypes.c_uint64,
                                       ctypes.c_int64, ctypes.c_int64, ctypes.c_int,
                                       ctypes.POINTER(_Opts), i32p]
        lib.oracle_run_ext.restype = ctypes.c_int
        lib.oracle_edges.argtypes = [ctypes.c_int, i32p, ctypes.c_int, i32p, i32p]
        lib.oracle_edges.restype = ctypes.c_int
        _lib = lib
        return lib


class _Opts(ctypes.Structure):
    _fields_ = [("opt", ctypes.c_int), ("beta1", ctypes.c_double), ("beta2", ctypes.c_double),
                ("eps", ctypes.c_double), ("drop", ctypes.POINTER(ctypes.c_uint8)),
                ("algo", ctypes.c_int), ("dme_count", ctypes.POINTER(ctypes.c_int64))]


ALGO_RELAYSGD, ALGO_GRAD, ALGO_DME = 0, 1, 2


OPT_SGD, OPT_NESTEROV, OPT_ADAM = 0, 1, 2


def _ptr(a: np.ndarray, ctype):
    return a.ctypes.data_as(ctypes.POINTER(ctype))


class OracleError(RuntimeError):
    def __init__(self, status: int):
        super().__init__(f"oracle returned status {status}")
        self.status = status


def _check(rc: int):
    if rc != ORACLE_OK:
        raise OracleError(rc)


def philox4x32_10(ctr, key) -> tuple:
    lib = _load()
    c = np.ascontiguousarray(np.asarray(ctr, dtype=np.uint32))
    k = np.ascontiguousarray(np.asarray(key, dtype=np.uint32))
    out = np.zeros(4, dtype=np.uint32)
    lib.oracle_philox4x32_10(_ptr(c, ctypes.c_uint32), _ptr(k, ctypes.c_uint32),
                             _ptr(out, ctypes.c_uint32))
    return tuple(int(v) for v in out)


def uniform(w: int) -> float:
    return _load().oracle_uniform(int(w) & 0xFFFFFFFF)


def normal(seed: int, c: int, row: int, step: int, stream: int) -> float:
    return _load().oracle_normal(seed, c, row, step, stream)


def normals(seed: int, c0: int, length: int, row: int, step: int, stream: int) -> np.ndarray:
    """oracle_normal for coordinates [c0, c0 + length) of (row, step, stream)."""
    lib = _load()
    out = np.zeros(max(length, 0), dtype=np.float64)
    _check(lib.oracle_fill_normals(seed, c0, length, row, step, stream, _ptr(out, ctypes.c_double)))
    return out


def _edges_arr(edges) -> np.ndarray:
    e = np.ascontiguousarray(np.asarray(edges, dtype=np.int32).reshape(-1, 2))
    return e


def edges(n: int, edge_list):
    """Directed-edge table (src, dst) of the oracle's own numbering."""
    lib = _load()
    e = _edges_arr(edge_list)
    E = 2 * e.shape[0]
    src = np.zeros(max(E, 1), dtype=np.int32)
    dst = np.zeros(max(E, 1), dtype=np.int32)
    _check(lib.oracle_edges(n, _ptr(e, ctypes.c_int32), e.shape[0],
                            _ptr(src, ctypes.c_int32), _ptr(dst, ctypes.c_int32)))
    return src[:E], dst[:E]


def fill_mu(n: int, mix: np.ndarray, mu_scale: float, seed: int, c0: int, length: int) -> np.ndarray:
    """mu_i(c) = mu_scale * sum_k mix[i, k] N_k(c) on coordinates [c0, c0+length)."""
    lib = _load()
    mix = np.ascontiguousarray(np.asarray(mix, dtype=np.float64).reshape(n, -1))
    K = mix.shape[1]
    mu = np.zeros((n, length), dtype=np.float64)
    _check(lib.oracle_fill_mu(n, K, _ptr(mix, ctypes.c_double), float(mu_scale), seed, c0,
                              length, _ptr(mu, ctypes.c_double)))
    return mu


def fill_x0(n: int, x0_std: float, seed: int, c0: int, length: int) -> np.ndarray:
    lib = _load()
    x = np.zeros((n, length), dtype=np.float64)
    _check(lib.oracle_fill_x0(n, float(x0_std), seed, c0, length, _ptr(x, ctypes.c_double)))
    return x


def run(n: int, edge_list, x: np.ndarray, mu: np.ndarray, msg: np.ndarray, counts: np.ndarray,
        lr: float, sigma: float, seed: int, step0: int, steps: int, mode: int = 0, c0: int = 0):
    """Runs ``steps`` iterations of Algorithm 1 in place on a coordinate slice.

    ``x``/``mu`` are [n][len], ``msg`` is [E][len] (m^{step0-1} in, the last
    m out), ``counts`` is int32[E] (c^{step0-1} in, the last c out).  Returns
    nbar^{step0+steps} as an int32[n] array.
    """
    lib = _load()
    e = _edges_arr(edge_list)
    E = 2 * e.shape[0]
    length = x.shape[1] if x.ndim == 2 else 0
    for a, rows in ((x, n), (mu, n), (msg, E)):
        assert a.dtype == np.float64 and a.flags.c_contiguous
        assert a.shape == (rows, length), (a.shape, rows, length)
    assert counts.dtype == np.int32 and counts.shape == (E,)
    nbar = np.zeros(n, dtype=np.int32)
    msg_p = msg if E > 0 else np.zeros((1, max(length, 1)))
    cnt_p = counts if E > 0 else np.zeros(1, dtype=np.int32)
    _check(lib.oracle_run(n, _ptr(e, ctypes.c_int32), e.shape[0], c0, length,
                          _ptr(x, ctypes.c_double), _ptr(mu, ctypes.c_double),
                          _ptr(msg_p, ctypes.c_double), _ptr(cnt_p, ctypes.c_int32),
                          float(lr), float(sigma), seed, step0, steps, mode,
                          _ptr(nbar, ctypes.c_int32)))
    return nbar


def run_ext(n: int, edge_list, x, mu, msg, counts, lr: float, sigma: float, seed: int,
            step0: int, steps: int, mode: int = 0, c0: int = 0, opt: int = OPT_SGD,
            beta1: float = 0.0, beta2: float = 0.0, eps: float = 0.0, s1=None, s2=None,
            drop=None, algo: int = ALGO_RELAYSGD, dme_count=None):
    """run() with a local optimiser (SGD / Nesterov momentum / Adam, state
    arrays s1, s2 [n][len] in place) and an optional mask drop[steps][E] of
    lost messages."""
    lib = _load()
    e = _edges_arr(edge_list)
    E = 2 * e.shape[0]
    length = x.shape[1]
    for a, rows in ((x, n), (mu, n), (msg, E)):
        assert a.dtype == np.float64 and a.flags.c_contiguous and a.shape == (rows, length)
    for a in (s1, s2):
        if a is not None:
            assert a.dtype == np.float64 and a.flags.c_contiguous and a.shape == (n, length)
    assert counts.dtype == np.int32 and counts.shape == (E,)
    o = _Opts(opt, beta1, beta2, eps, None, algo, None)
    if algo == ALGO_DME:
        assert dme_count is not None and dme_count.dtype == np.int64 and dme_count.shape == (n,)
        o.dme_count = dme_count.ctypes.data_as(ctypes.POINTER(ctypes.c_int64))
    if drop is not None:
        drop = np.ascontiguousarray(np.asarray(drop, dtype=np.uint8).reshape(steps, E))
        o.drop = drop.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8))
    nbar = np.zeros(n, dtype=np.int32)
    msg_p = msg if E > 0 else np.zeros((1, max(length, 1)))
    cnt_p = counts if E > 0 else np.zeros(1, dtype=np.int32)
    null = ctypes.POINTER(ctypes.c_double)()
    _check(lib.oracle_run_ext(n, _ptr(e, ctypes.c_int32), e.shape[0], c0, length,
                              _ptr(x, ctypes.c_double), _ptr(mu, ctypes.c_double),
                              _ptr(msg_p, ctypes.c_double), _ptr(cnt_p, ctypes.c_int32),
                              _ptr(s1, ctypes.c_double) if s1 is not None else null,
                              _ptr(s2, ctypes.c_double) if s2 is not None else null,
                              float(lr), float(sigma), seed, step0, steps, mode, ctypes.byref(o),
                              _ptr(nbar, ctypes.c_int32)))
    return nbar


class State:
    """Oracle-side state of a RelaySum run on coordinate slice [c0, c0+len)."""

    def __init__(self, n: int, edge_list, length: int, c0: int = 0):
        self.n = n
        self.edges = _edges_arr(edge_list)
        self.E = 2 * self.edges.shape[0]
        self.c0 = c0
        self.length = length
        self.x = np.zeros((n, length))
        self.mu = np.zeros((n, length))
        self.msg = np.zeros((self.E, length))
        self.counts = np.zeros(self.E, dtype=np.int32)
        self.step = 0

    def init(self, x0_std: float, seed: int, mix=None, mu_scale: float = 0.0, mu_seed: int = 0):
        self.x = fill_x0(self.n, x0_std, seed, self.c0, self.length)
        if mix is not None:
            self.mu = fill_mu(self.n, mix, mu_scale, mu_seed, self.c0, self.length)
        self.msg[:] = 0.0
        self.counts[:] = 0
        self.step = 0
        self.s1 = np.zeros((self.n, self.length))
        self.s2 = np.zeros((self.n, self.length))
        self.dme_count = np.zeros(self.n, dtype=np.int64)

    def advance(self, steps: int, lr: float, sigma: float, seed: int, mode: int = 0,
                opt: int = OPT_SGD, beta1: float = 0.0, beta2: float = 0.0, eps: float = 0.0,
                drop=None, algo: int = ALGO_RELAYSGD):
        if not hasattr(self, "dme_count"):
            self.dme_count = np.zeros(self.n, dtype=np.int64)
        if opt == OPT_SGD and drop is None and algo == ALGO_RELAYSGD:
            nbar = run(self.n, self.edges, self.x, self.mu, self.msg, self.counts, lr, sigma,
                       seed, self.step, steps, mode, self.c0)
        else:
            if not hasattr(self, "s1"):
                self.s1 = np.zeros((self.n, self.length))
                self.s2 = np.zeros((self.n, self.length))
            nbar = run_ext(self.n, self.edges, self.x, self.mu, self.msg, self.counts, lr, sigma,
                           seed, self.step, steps, mode, self.c0, opt, beta1, beta2, eps,
                           self.s1, self.s2, drop, algo, self.dme_count)
        self.step += steps
        return nbar
