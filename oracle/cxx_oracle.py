"""ctypes binding of the C++ oracle (oracle/dsm_oracle.cpp).

TEST INFRASTRUCTURE.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference arms of ``bench.py`` may import this module.  It
loads ``libdsm_oracle.so`` (built here from ``dsm_oracle.cpp`` with g++,
``-O2 -ffp-contract=off``, OpenMP over elements), never the CUDA library.

:class:`CxxOracleRun` has the interface of the numpy oracle's ``OracleRun``
(x, m, X, opt_m, opt_v, gv, t, k, gamma, last_stats, last_inter;
local_step, global_step, run_round) and computes the same values bit for
bit: one global round of Algorithm 1 of arXiv 2411.17866 on any subset of
element indices.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from ctypes import POINTER, c_float, c_int, c_int32, c_int64, c_uint32, c_uint64, c_void_p

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "dsm_oracle.cpp")
LIB = os.path.join(HERE, "libdsm_oracle.so")
# No contraction and no fast-math: one IEEE rounding per operation, as the paper's expressions are written.
CXX_FLAGS = ["-O2", "-std=c++17", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared"]

FLAG_RESET_LOCAL_STATE = 2
GLOBAL_ADAMW = 4


class dsmo_tensor(ctypes.Structure):
    _fields_ = [("numel", c_uint64), ("grad_scale", c_float), ("kind", c_uint32), ("wd", c_uint32)]


class dsmo_hparams(ctypes.Structure):
    _fields_ = [("base", c_int32), ("lr", c_float), ("b1", c_float), ("b2", c_float), ("eps", c_float),
                ("wd", c_float), ("mu", c_float), ("g_b1", c_float), ("g_b2", c_float), ("g_eta", c_float),
                ("g_wd", c_float), ("sign_mode", c_int32), ("rsign_B", c_float), ("grad_dtype", c_int32),
                ("flags", c_uint32), ("seed", c_uint64), ("global_mode", c_int32), ("g_eps", c_float)]


class dsmo_stats(ctypes.Structure):
    _fields_ = [("delta_sq", ctypes.c_double), ("drift", ctypes.c_double), ("zero_sign", c_uint64),
                ("flips", c_uint64), ("unanimous", c_uint64), ("clamped", c_uint64)]

    def as_dict(self):
        return {f: (float(getattr(self, f)) if f in ("delta_sq", "drift") else int(getattr(self, f)))
                for f, _ in self._fields_}


def build(verbose: bool = False, out: str = LIB) -> str:
    """Compile libdsm_oracle.so with g++ (OpenMP if the compiler has it)."""
    tmp = out + ".tmp"
    last = None
    for extra in (["-fopenmp"], ["-Wno-unknown-pragmas"]):
        cmd = ["g++", *CXX_FLAGS, *extra, "-o", tmp, SRC]
        if verbose:
            print(" ".join(cmd), flush=True)
        r = subprocess.run(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
        if r.returncode == 0:
            os.replace(tmp, out)
            return out
        last = r.stdout
    raise RuntimeError(f"building the C++ oracle failed:\n{last}")


_lib = None


def load() -> ctypes.CDLL:
    """The oracle library, built first if it is missing or older than its source."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB) or os.path.getmtime(LIB) < os.path.getmtime(SRC):
        build()
    lib = ctypes.CDLL(LIB)
    fp = POINTER(c_float)
    lib.dsmo_create.restype = c_void_p
    lib.dsmo_create.argtypes = [POINTER(dsmo_tensor), c_uint32, c_uint32, POINTER(dsmo_hparams), POINTER(c_int64),
                                c_uint64, c_uint64, c_int]
    lib.dsmo_destroy.argtypes = [c_void_p]
    lib.dsmo_init_x0.argtypes = [c_void_p, fp]
    lib.dsmo_synthetic_grad.argtypes = [c_void_p, c_uint64, c_uint32, fp]
    lib.dsmo_local_step.argtypes = [c_void_p, fp, fp, fp, fp, c_uint64, c_uint64, c_float]
    lib.dsmo_global_step.argtypes = [c_void_p, fp, fp, fp, fp, c_float, c_uint64, POINTER(dsmo_stats), fp, fp, fp,
                                     fp, fp]
    lib.dsmo_splitmix64_output.restype = c_uint64
    lib.dsmo_splitmix64_output.argtypes = [c_uint64, c_uint64]
    lib.dsmo_philox4x32_10.argtypes = [POINTER(c_uint32), POINTER(c_uint32), POINTER(c_uint32)]
    lib.dsmo_philox_uniform.restype = c_float
    lib.dsmo_philox_uniform.argtypes = [c_uint64, c_uint64, c_uint64]
    lib.dsmo_uniform24.restype = c_float
    lib.dsmo_uniform24.argtypes = [c_uint64, c_uint64, c_uint64, c_uint64]
    lib.dsmo_bf16_round.restype = c_float
    lib.dsmo_bf16_round.argtypes = [c_float]
    lib.dsmo_max_threads.restype = c_int
    _lib = lib
    return lib


def _fptr(a):
    return None if a is None else a.ctypes.data_as(POINTER(c_float))


def make_hparams(hp) -> dsmo_hparams:
    h = dsmo_hparams()
    defaults = {"global_mode": 0, "g_eps": 1e-8, "flags": 0}
    for name, _ in dsmo_hparams._fields_:
        setattr(h, name, getattr(hp, name, defaults.get(name)))
    return h


def splitmix64_output(state: int, j: int) -> int:
    return int(load().dsmo_splitmix64_output(state, j))


def philox4x32_10(ctr, key):
    c = (c_uint32 * 4)(*ctr)
    k = (c_uint32 * 2)(*key)
    out = (c_uint32 * 4)()
    load().dsmo_philox4x32_10(c, k, out)
    return [int(v) for v in out]


def philox_uniform(seed: int, t: int, e: int) -> float:
    return float(load().dsmo_philox_uniform(seed, t, e))


def uniform24(seed: int, stream: int, idx: int, e: int) -> float:
    return float(load().dsmo_uniform24(seed, stream, idx, e))


def bf16_round(v: float) -> float:
    return float(load().dsmo_bf16_round(v))


class CxxOracleRun:
    """Algorithm 1 over a set of elements of one parameter layout, computed by the C++ oracle.

    Same arguments and attributes as the numpy oracle's OracleRun (float32 only, first_element
    included), plus ``threads`` (0: OpenMP's default).  X, opt_m and opt_v are [n][count] arrays (row i is worker i).
    """

    def __init__(self, tensors, n, tau, hp, elems=None, x0=None, with_stats=False, threads=0, first_element=0):
        lib = load()
        self.tensors = list(tensors)
        self.n, self.tau, self.hp = int(n), int(tau), hp
        self.d = int(sum(t.numel for t in self.tensors))
        self.elems = np.ascontiguousarray(np.arange(self.d, dtype=np.int64) if elems is None else elems,
                                          dtype=np.int64)
        self.count = int(self.elems.size)
        arr = (dsmo_tensor * len(self.tensors))()
        for i, t in enumerate(self.tensors):
            arr[i].numel, arr[i].grad_scale = int(t.numel), float(t.grad_scale)
            arr[i].kind, arr[i].wd = int(t.kind), int(getattr(t, "wd", 1))
        self._hp = make_hparams(hp)
        self._ctx = lib.dsmo_create(arr, len(self.tensors), self.n, ctypes.byref(self._hp),
                                    self.elems.ctypes.data_as(POINTER(c_int64)), self.count, int(first_element),
                                    int(threads))
        if not self._ctx:
            raise ValueError("an element index lies outside the model")
        self.x = np.empty(self.count, dtype=np.float32)
        if x0 is None:
            lib.dsmo_init_x0(self._ctx, _fptr(self.x))
        else:
            self.x[:] = np.asarray(x0, dtype=np.float32)
        self.m = np.zeros(self.count, dtype=np.float32)
        self.X = np.tile(self.x, (self.n, 1))
        self.opt_m = np.zeros((self.n, self.count), dtype=np.float32)
        self.opt_v = np.zeros((self.n, self.count), dtype=np.float32) if hp.base == 0 else None
        self.global_mode = getattr(hp, "global_mode", 0)
        self.gv = np.zeros(self.count, dtype=np.float32) if self.global_mode == GLOBAL_ADAMW else None
        self.reset_local = bool(getattr(hp, "flags", 0) & FLAG_RESET_LOCAL_STATE)
        self.t = 0
        self.k = 0
        self.gamma = hp.lr
        self.with_stats = with_stats
        self.last_stats = None
        self.last_inter = None

    def __del__(self):
        ctx, self._ctx = getattr(self, "_ctx", None), None
        if ctx and _lib is not None:
            _lib.dsmo_destroy(ctx)

    def grads(self, step: int, worker: int) -> np.ndarray:
        g = np.empty(self.count, dtype=np.float32)
        load().dsmo_synthetic_grad(self._ctx, step, worker, _fptr(g))
        return g

    def local_step(self, grads=None):
        """Local step k of the current round for every worker, Eq. (local-steps)."""
        assert self.k < self.tau
        step = self.t * self.tau + self.k
        j = self.k + 1 if self.reset_local else step + 1
        g = None
        if grads is not None:
            g = np.ascontiguousarray(np.stack([np.asarray(gi, dtype=np.float32) for gi in grads]))
            assert g.shape == (self.n, self.count)
        load().dsmo_local_step(self._ctx, _fptr(self.X), _fptr(self.opt_m), _fptr(self.opt_v), _fptr(g), step, j,
                               float(self.gamma))
        self.k += 1

    def global_step(self, r=None, lam=None):
        """All-reduce average, sign-momentum (or ablation) update and synchronisation (Algorithm 1).
        ``r`` and ``lam`` optionally give the randomized sign's uniforms and the per-element decay."""
        assert self.k == self.tau
        stats = (dsmo_stats * len(self.tensors))() if self.with_stats else None
        delta, u, sg = (np.empty(self.count, dtype=np.float32) for _ in range(3))
        r = None if r is None else np.ascontiguousarray(r, dtype=np.float32)
        lam = None if lam is None else np.ascontiguousarray(lam, dtype=np.float32)
        load().dsmo_global_step(self._ctx, _fptr(self.x), _fptr(self.m), _fptr(self.gv), _fptr(self.X),
                                float(self.gamma), self.t, stats, _fptr(delta), _fptr(u), _fptr(sg), _fptr(r),
                                _fptr(lam))
        self.last_stats = [s.as_dict() for s in stats] if stats is not None else None
        self.last_inter = {"delta": delta, "u": u, "sg": sg}
        if self.reset_local:
            self.opt_m[:] = 0
            if self.opt_v is not None:
                self.opt_v[:] = 0
        self.t += 1
        self.k = 0

    def run_round(self, grads=None):
        """One global round; ``grads`` optionally gives grads[k][i] explicitly."""
        for k in range(self.tau):
            self.local_step(None if grads is None else grads[k])
        self.global_step()
