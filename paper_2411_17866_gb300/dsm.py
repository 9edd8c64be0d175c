"""Python binding of libdsm.so (include/dsm.h): argument marshalling only.

Each ``dsm_*`` function here calls the C function of the same name through
ctypes and raises :class:`DsmError` on a negative return code.  Every step
of the method runs in the library's CUDA kernels; PyTorch only supplies the
device memory (the arena, a uint8 tensor) and the current CUDA stream.

:class:`DistributedSignMomentum` is a thin convenience wrapper that owns the
arena tensor and a handle and exposes the round as Python methods.
"""
from __future__ import annotations

import collections
import ctypes
import math
import os
from ctypes import POINTER, byref, c_char_p, c_float, c_int, c_int32, c_size_t, c_uint32, c_uint64, c_void_p

_HERE = os.path.dirname(os.path.abspath(__file__))
# The in-tree library; DSM_LIBRARY may name another build of it (e.g. the contracting release build).
LIB_PATH = os.environ.get("DSM_LIBRARY") or os.path.join(_HERE, "libdsm.so")

DSM_OK, DSM_EINVAL, DSM_ENOMEM, DSM_EALIGN, DSM_ESTATE, DSM_ECUDA, DSM_ERANGE = 0, -1, -2, -3, -4, -5, -6
KIND_WEIGHT, KIND_BIAS, KIND_LN_W, KIND_LN_B = 0, 1, 2, 3
BASE_ADAMW, BASE_SGDM = 0, 1
SIGN, RSIGN_ZERO, RSIGN_PM = 0, 1, 2
F32, BF16 = 0, 1
BUF_X, BUF_M, BUF_REPLICA, BUF_OPT_M, BUF_OPT_V, BUF_GRAD, BUF_GLOBAL_V = 0, 1, 2, 3, 4, 5, 6
GLOBAL_SIGN_MOMENTUM, GLOBAL_SLOWMO, GLOBAL_SIGNED_SLOWMO, GLOBAL_LOOKAHEAD, GLOBAL_ADAMW = 0, 1, 2, 3, 4
FLAG_FUSED_ROUND = 1
FLAG_RESET_LOCAL_STATE = 2

ERROR_NAMES = {DSM_EINVAL: "DSM_EINVAL", DSM_ENOMEM: "DSM_ENOMEM", DSM_EALIGN: "DSM_EALIGN",
               DSM_ESTATE: "DSM_ESTATE", DSM_ECUDA: "DSM_ECUDA", DSM_ERANGE: "DSM_ERANGE"}


class DsmError(RuntimeError):
    def __init__(self, code: int, func: str, msg: str):
        super().__init__(f"{func} failed with {ERROR_NAMES.get(code, code)}: {msg}")
        self.code = code


class dsm_tensor(ctypes.Structure):
    _fields_ = [("numel", c_uint64), ("grad_scale", c_float), ("kind", c_uint32), ("wd", c_uint32),
                ("reserved", c_uint32)]


class dsm_layout(ctypes.Structure):
    _fields_ = [("tensors", POINTER(dsm_tensor)), ("count", c_uint32), ("first_element", c_uint64)]


class dsm_hparams(ctypes.Structure):
    _fields_ = [("base", c_int32), ("lr", c_float), ("b1", c_float), ("b2", c_float), ("eps", c_float),
                ("wd", c_float), ("mu", c_float), ("g_b1", c_float), ("g_b2", c_float), ("g_eta", c_float),
                ("g_wd", c_float), ("sign_mode", c_int32), ("rsign_B", c_float), ("grad_dtype", c_int32),
                ("flags", c_uint32), ("seed", c_uint64), ("global_mode", c_int32), ("g_eps", c_float)]


class dsm_tensor_stats(ctypes.Structure):
    _fields_ = [("delta_sq", ctypes.c_double), ("drift", ctypes.c_double), ("zero_sign", c_uint64),
                ("flips", c_uint64), ("unanimous", c_uint64), ("clamped", c_uint64)]

    def as_dict(self):
        return {f: getattr(self, f) for f, _ in self._fields_}


class dsm_info(ctypes.Structure):
    _fields_ = [("d", c_uint64), ("d_stride", c_uint64), ("n", c_uint32), ("tau", c_uint32),
                ("num_tensors", c_uint32), ("num_tiles", c_uint32), ("round", c_uint64),
                ("local_steps", c_uint32), ("gamma", c_float)]


_PROTOS = {
    "dsm_state_bytes": (c_size_t, [POINTER(dsm_layout), c_uint32, POINTER(dsm_hparams)]),
    "dsm_create": (c_int, [POINTER(dsm_layout), c_uint32, c_uint32, POINTER(dsm_hparams), c_void_p, c_size_t,
                           c_void_p, c_int, c_void_p, POINTER(c_void_p)]),
    "dsm_set_gamma": (c_int, [c_void_p, c_float]),
    "dsm_fill_synthetic_grads": (c_int, [c_void_p, c_uint64, c_void_p]),
    "dsm_grad_ptr": (c_int, [c_void_p, c_uint32, POINTER(c_void_p)]),
    "dsm_replica_ptr": (c_int, [c_void_p, c_uint32, c_void_p, POINTER(c_void_p)]),
    "dsm_load_grads": (c_int, [c_void_p, c_void_p, c_int, c_void_p]),
    "dsm_local_step": (c_int, [c_void_p, c_void_p]),
    "dsm_local_step_host_grads": (c_int, [c_void_p, c_void_p, c_void_p, c_void_p]),
    "dsm_global_step": (c_int, [c_void_p, c_void_p, POINTER(dsm_tensor_stats), c_uint32]),
    "dsm_stats_ptr": (c_int, [c_void_p, POINTER(c_void_p)]),
    "dsm_read_params": (c_int, [c_void_p, c_int, c_uint32, c_void_p, c_uint64, c_uint64, c_int, c_void_p]),
    "dsm_write_params": (c_int, [c_void_p, c_int, c_uint32, c_void_p, c_uint64, c_uint64, c_int, c_void_p]),
    "dsm_set_round": (c_int, [c_void_p, c_uint64]),
    "dsm_set_first_worker": (c_int, [c_void_p, c_uint32]),
    "dsm_end_round": (c_int, [c_void_p, c_void_p, c_int, c_void_p]),
    "dsm_cosine_gamma": (c_int, [c_float, c_float, c_uint64, c_uint64, c_uint64, POINTER(c_float)]),
    "dsm_get_info": (c_int, [c_void_p, POINTER(dsm_info)]),
    "dsm_check_guards": (c_int, [c_void_p, c_void_p, POINTER(c_uint32)]),
    "dsm_destroy": (c_int, [c_void_p]),
    "dsm_last_error": (c_char_p, []),
    "dsm_global_step_noalloc": (c_int, [POINTER(dsm_layout), c_uint32, POINTER(dsm_hparams), c_float, c_uint64,
                                        c_void_p, c_void_p, c_void_p, c_uint64, POINTER(dsm_tensor_stats), c_int,
                                        c_void_p]),
}

_lib = None


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libdsm.so; raises if it has not been built (there is no fallback)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'` "
                           "(the CUDA library is required; there is no CPU fallback)")
    lib = ctypes.CDLL(path)
    for name, (res, args) in _PROTOS.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def last_error() -> str:
    return load_library().dsm_last_error().decode()


def _check(rc: int, func: str) -> None:
    if rc != DSM_OK:
        raise DsmError(rc, func, last_error())


def _stream(stream) -> c_void_p:
    """A cudaStream_t from a torch stream, an int handle, or None (torch's current stream)."""
    if stream is None:
        import torch
        return c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return c_void_p(stream)
    return c_void_p(stream.cuda_stream)


def make_layout(tensors, first_element: int = 0):
    """A dsm_layout from objects with numel, grad_scale, kind and wd; keep the result alive while used.
    first_element: the layout's first element within a larger model (a parameter shard), else 0."""
    arr = (dsm_tensor * len(tensors))()
    for i, t in enumerate(tensors):
        arr[i].numel = int(t.numel)
        arr[i].grad_scale = float(t.grad_scale)
        arr[i].kind = int(t.kind)
        arr[i].wd = int(getattr(t, "wd", 1))
        arr[i].reserved = 0
    lay = dsm_layout(ctypes.cast(arr, POINTER(dsm_tensor)), len(tensors), int(first_element))
    lay._keep = arr
    return lay


LayoutEntry = collections.namedtuple("LayoutEntry", "numel grad_scale kind wd")


def make_hparams(hp) -> dsm_hparams:
    """A dsm_hparams from an object with the same field names."""
    h = dsm_hparams()
    defaults = {"global_mode": 0, "g_eps": 1e-8, "flags": 0}
    for name, _ in dsm_hparams._fields_:
        setattr(h, name, getattr(hp, name, defaults.get(name)))
    return h


# ---- the C functions, same names ----------------------------------------

def dsm_state_bytes(layout: dsm_layout, n: int, hp: dsm_hparams) -> int:
    nb = load_library().dsm_state_bytes(byref(layout), n, byref(hp))
    if nb == 0:
        raise DsmError(DSM_EINVAL, "dsm_state_bytes", last_error())
    return nb


def dsm_create(layout, n, tau, hp, arena_ptr: int, arena_bytes: int, x0_ptr=None, x0_is_device=False,
               stream=None) -> c_void_p:
    h = c_void_p()
    rc = load_library().dsm_create(byref(layout), n, tau, byref(hp), c_void_p(arena_ptr), arena_bytes,
                                   c_void_p(x0_ptr) if x0_ptr else None, int(bool(x0_is_device)),
                                   _stream(stream), byref(h))
    _check(rc, "dsm_create")
    return h


def dsm_set_gamma(h, gamma: float) -> None:
    _check(load_library().dsm_set_gamma(h, gamma), "dsm_set_gamma")


def dsm_fill_synthetic_grads(h, step: int, stream=None) -> None:
    _check(load_library().dsm_fill_synthetic_grads(h, step, _stream(stream)), "dsm_fill_synthetic_grads")


def dsm_grad_ptr(h, worker: int) -> int:
    p = c_void_p()
    _check(load_library().dsm_grad_ptr(h, worker, byref(p)), "dsm_grad_ptr")
    return p.value


def dsm_replica_ptr(h, worker: int, stream=None) -> int:
    p = c_void_p()
    _check(load_library().dsm_replica_ptr(h, worker, _stream(stream), byref(p)), "dsm_replica_ptr")
    return p.value


def dsm_load_grads(h, src_ptr: int, src_is_device: bool, stream=None) -> None:
    _check(load_library().dsm_load_grads(h, c_void_p(src_ptr), int(bool(src_is_device)), _stream(stream)),
           "dsm_load_grads")


def dsm_local_step(h, stream=None) -> None:
    _check(load_library().dsm_local_step(h, _stream(stream)), "dsm_local_step")


def dsm_local_step_host_grads(h, src_ptr: int, stream=None, copy_stream=None) -> None:
    """``copy_stream``: the stream for the chunked host-to-device copies (None: ``stream``)."""
    cs = _stream(stream) if copy_stream is None else _stream(copy_stream)
    _check(load_library().dsm_local_step_host_grads(h, c_void_p(src_ptr), _stream(stream), cs),
           "dsm_local_step_host_grads")


def dsm_global_step(h, stream=None, stats=None) -> None:
    """``stats``: None, or a ctypes array of dsm_tensor_stats (host) to fill (synchronises)."""
    if stats is None:
        rc = load_library().dsm_global_step(h, _stream(stream), None, 0)
    else:
        rc = load_library().dsm_global_step(h, _stream(stream), ctypes.cast(stats, POINTER(dsm_tensor_stats)),
                                            len(stats))
    _check(rc, "dsm_global_step")


def dsm_stats_ptr(h) -> int:
    p = c_void_p()
    _check(load_library().dsm_stats_ptr(h, byref(p)), "dsm_stats_ptr")
    return p.value


def dsm_read_params(h, which: int, worker: int, dst_ptr: int, offset: int, count: int, dst_is_device: bool,
                    stream=None) -> None:
    _check(load_library().dsm_read_params(h, which, worker, c_void_p(dst_ptr), offset, count,
                                          int(bool(dst_is_device)), _stream(stream)), "dsm_read_params")


def dsm_write_params(h, which: int, worker: int, src_ptr: int, offset: int, count: int, src_is_device: bool,
                     stream=None) -> None:
    _check(load_library().dsm_write_params(h, which, worker, c_void_p(src_ptr), offset, count,
                                           int(bool(src_is_device)), _stream(stream)), "dsm_write_params")


def dsm_set_round(h, round_: int) -> None:
    _check(load_library().dsm_set_round(h, round_), "dsm_set_round")


def dsm_set_first_worker(h, first_worker: int) -> None:
    _check(load_library().dsm_set_first_worker(h, first_worker), "dsm_set_first_worker")


def dsm_end_round(h, x_ptr: int, x_is_device: bool, stream=None) -> None:
    _check(load_library().dsm_end_round(h, c_void_p(x_ptr), int(bool(x_is_device)), _stream(stream)),
           "dsm_end_round")


def dsm_cosine_gamma(peak: float, final_ratio: float, warmup_steps: int, total_steps: int, step: int) -> float:
    out = c_float()
    _check(load_library().dsm_cosine_gamma(peak, final_ratio, warmup_steps, total_steps, step, byref(out)),
           "dsm_cosine_gamma")
    return out.value


def dsm_get_info(h) -> dsm_info:
    info = dsm_info()
    _check(load_library().dsm_get_info(h, byref(info)), "dsm_get_info")
    return info


def dsm_check_guards(h, stream=None) -> int:
    """Number of arena guard regions that a write past the end of a buffer changed (0 = intact)."""
    bad = c_uint32()
    _check(load_library().dsm_check_guards(h, _stream(stream), byref(bad)), "dsm_check_guards")
    return bad.value


def dsm_destroy(h) -> None:
    _check(load_library().dsm_destroy(h), "dsm_destroy")


def dsm_global_step_noalloc(layout, n, hp, gamma, round_, x_ptr, m_ptr, replicas_ptr, replica_stride,
                            stats=None, stats_is_device=False, stream=None) -> None:
    """The global step on caller-owned device buffers, with the library's static scratch array
    (for callers that cannot allocate device memory).  ``stats``: None, a ctypes array of
    dsm_tensor_stats in host memory, or a device address (int) with stats_is_device=True."""
    if stats is None:
        sp = None
    elif stats_is_device:
        sp = ctypes.cast(c_void_p(stats), POINTER(dsm_tensor_stats))
    else:
        sp = ctypes.cast(stats, POINTER(dsm_tensor_stats))
    rc = load_library().dsm_global_step_noalloc(byref(layout), n, byref(hp), gamma, round_, c_void_p(x_ptr),
                                                c_void_p(m_ptr), c_void_p(replicas_ptr), replica_stride, sp,
                                                int(bool(stats_is_device)), _stream(stream))
    _check(rc, "dsm_global_step_noalloc")


# ---- convenience wrapper --------------------------------------------------

class DistributedSignMomentum:
    """One problem instance: the arena (a torch uint8 tensor on ``device``) and its handle.

    tensors: objects with numel, grad_scale, kind, wd; hp: an object with
    the dsm_hparams field names.  x0: optional float32 torch tensor of d
    elements (host or device).  first_element: where this layout starts in a
    larger model of which it is a parameter shard (dsm_layout.first_element).
    """

    shapes = None   # the tensors' shapes, for a problem built by from_tensors

    def __init__(self, tensors, n: int, tau: int, hp, device="cuda", x0=None, stream=None, first_element: int = 0):
        import torch
        self.layout = make_layout(tensors, first_element)
        self.hp = make_hparams(hp)
        self.n, self.tau = int(n), int(tau)
        self.nbytes = dsm_state_bytes(self.layout, self.n, self.hp)
        self.device = torch.device(device)
        raw = torch.empty(self.nbytes + 256, dtype=torch.uint8, device=self.device)
        shift = (-raw.data_ptr()) % 256
        self.arena = raw[shift:shift + self.nbytes]
        self._raw = raw
        x0_ptr, x0_dev = None, False
        if x0 is not None:
            x0 = x0.contiguous().to(torch.float32)
            self._x0 = x0
            x0_ptr, x0_dev = x0.data_ptr(), x0.is_cuda
        with torch.cuda.device(self.device):
            self.h = dsm_create(self.layout, self.n, self.tau, self.hp, self.arena.data_ptr(), self.nbytes,
                                x0_ptr, x0_dev, stream)
        info = dsm_get_info(self.h)
        self.d, self.d_stride = int(info.d), int(info.d_stride)
        self.num_tensors = int(info.num_tensors)

    @classmethod
    def from_tensors(cls, params, n: int, tau: int, hp, device="cuda", decay=None, stream=None):
        """A problem over the given tensors (e.g. a torch module's parameters, in order): one layout
        entry per tensor (kind weight for tensors of two or more dimensions, bias otherwise; decoupled
        weight decay on every tensor unless ``decay``, one bool per tensor, says otherwise), and the
        initial model x0 = their current values, concatenated.  ``unflatten`` splits a flat buffer
        back into tensors of these shapes."""
        import torch
        params = [p.detach() for p in params]
        decay = [True] * len(params) if decay is None else list(decay)
        if len(decay) != len(params):
            raise ValueError("decay needs one entry per tensor")
        layout = [LayoutEntry(int(p.numel()), 0.0, KIND_WEIGHT if p.dim() >= 2 else KIND_BIAS, int(bool(wd)))
                  for p, wd in zip(params, decay)]
        x0 = torch.cat([p.reshape(-1).to(torch.float32) for p in params]).to(device)
        obj = cls(layout, n, tau, hp, device=device, x0=x0, stream=stream)
        obj.shapes = [tuple(p.shape) for p in params]
        return obj

    def unflatten(self, flat):
        """Views of a flat d-element tensor (a replica, x, a gradient buffer) shaped like the tensors
        given to from_tensors."""
        if self.shapes is None:
            raise ValueError("unflatten needs a problem built by from_tensors")
        out, off = [], 0
        for shape in self.shapes:
            k = math.prod(shape)
            out.append(flat[off:off + k].view(shape))
            off += k
        return out

    # Algorithm 1, one call per step
    def set_gamma(self, gamma):
        dsm_set_gamma(self.h, gamma)

    def fill_synthetic_grads(self, step, stream=None):
        dsm_fill_synthetic_grads(self.h, step, stream)

    def set_first_worker(self, first_worker):
        """Worker i draws the synthetic gradients of worker first_worker + i of a larger set."""
        dsm_set_first_worker(self.h, first_worker)

    def load_grads(self, src, stream=None):
        dsm_load_grads(self.h, src.data_ptr(), src.is_cuda, stream)

    def local_step(self, stream=None):
        dsm_local_step(self.h, stream)

    def _arena_view(self, ptr: int, count: int, dtype):
        """A tensor aliasing `count` elements of the arena at device address `ptr`."""
        import torch
        esize = torch.tensor([], dtype=dtype).element_size()
        off = ptr - self.arena.data_ptr()
        if off < 0 or off + count * esize > self.nbytes:
            raise DsmError(DSM_ERANGE, "_arena_view", "address outside the arena")
        return self.arena[off:off + count * esize].view(dtype)

    def replica_view(self, worker, stream=None):
        """Worker `worker`'s current model x^(i) as a read-only-by-contract float32 CUDA tensor of d
        elements (aliasing the arena; valid until the next step or state write)."""
        import torch
        return self._arena_view(dsm_replica_ptr(self.h, worker, stream), self.d, torch.float32)

    def grad_view(self, worker):
        """Worker `worker`'s gradient buffer as a CUDA tensor of d elements of the gradient type
        (aliasing the arena), for a caller that writes its own gradients."""
        import torch
        dt = torch.bfloat16 if self.hp.grad_dtype == BF16 else torch.float32
        return self._arena_view(dsm_grad_ptr(self.h, worker), self.d, dt)

    def local_step_host_grads(self, src, stream=None, copy_stream=None):
        """One local step on gradients in host memory (``src``: [n, d] CPU tensor of the gradient type,
        pinned for overlap), the copy of each chunk overlapped with the update of the previous one."""
        esize = 2 if self.hp.grad_dtype == BF16 else 4
        if src.is_cuda or not src.is_contiguous() or tuple(src.shape) != (self.n, self.d) or \
                src.element_size() != esize:
            raise ValueError(f"src must be a contiguous [n, d] host tensor of {esize}-byte gradients")
        dsm_local_step_host_grads(self.h, src.data_ptr(), stream, copy_stream)

    def global_step(self, stream=None, with_stats=False):
        if not with_stats:
            dsm_global_step(self.h, stream)
            return None
        arr = (dsm_tensor_stats * self.num_tensors)()
        dsm_global_step(self.h, stream, arr)
        return [a.as_dict() for a in arr]

    def end_round(self, x_next, stream=None):
        """End the round with a global model computed elsewhere (d fp32 values, CPU or CUDA tensor):
        every worker restarts from it and the round counter advances; no global step runs here."""
        import torch
        x_next = x_next.contiguous()
        if x_next.dtype != torch.float32 or x_next.numel() != self.d:
            raise ValueError(f"x_next must hold {self.d} float32 values")
        dsm_end_round(self.h, x_next.data_ptr(), x_next.is_cuda, stream)

    def synthetic_round(self, stream=None, with_stats=False):
        """tau x (synthetic gradients + local step), then the global step."""
        info = dsm_get_info(self.h)
        base = int(info.round) * self.tau
        for k in range(self.tau):
            self.fill_synthetic_grads(base + k, stream)
            self.local_step(stream)
        return self.global_step(stream, with_stats)

    def read(self, which, worker=0, offset=0, count=None, out=None, stream=None):
        """Buffer `which` as a tensor (a new CPU tensor unless ``out`` is given)."""
        import torch
        count = self.d - offset if count is None else count
        dt = torch.float32
        if which == BUF_GRAD and self.hp.grad_dtype == BF16:
            dt = torch.bfloat16
        if out is None:
            out = torch.empty(count, dtype=dt)
        dsm_read_params(self.h, which, worker, out.data_ptr(), offset, count, out.is_cuda, stream)
        return out

    def write(self, which, src, worker=0, offset=0, stream=None):
        src = src.contiguous()
        dsm_write_params(self.h, which, worker, src.data_ptr(), offset, src.numel(), src.is_cuda, stream)

    def info(self):
        return dsm_get_info(self.h)

    def check_guards(self, stream=None) -> int:
        return dsm_check_guards(self.h, stream)

    def state_dict(self) -> dict:
        """Every buffer of the method's state as CPU tensors, with the round counter and gamma_t
        (call between rounds).  Gradients are not part of the state."""
        info = dsm_get_info(self.h)
        if info.local_steps != 0:
            raise DsmError(DSM_ESTATE, "state_dict", "take a checkpoint between rounds")
        st = {"round": int(info.round), "gamma": float(info.gamma), "x": self.read(BUF_X), "m": self.read(BUF_M),
              "replicas": [self.read(BUF_REPLICA, i) for i in range(self.n)],
              "opt_m": [self.read(BUF_OPT_M, i) for i in range(self.n)]}
        if self.hp.base == BASE_ADAMW:
            st["opt_v"] = [self.read(BUF_OPT_V, i) for i in range(self.n)]
        if self.hp.global_mode == GLOBAL_ADAMW:
            st["global_v"] = self.read(BUF_GLOBAL_V)
        return st

    def load_state_dict(self, st: dict) -> None:
        """Restore a state_dict() into this handle (same layout, n and hyper-parameters)."""
        self.write(BUF_X, st["x"])
        self.write(BUF_M, st["m"])
        for i in range(self.n):
            self.write(BUF_REPLICA, st["replicas"][i], worker=i)
            self.write(BUF_OPT_M, st["opt_m"][i], worker=i)
            if "opt_v" in st:
                self.write(BUF_OPT_V, st["opt_v"][i], worker=i)
        if "global_v" in st:
            self.write(BUF_GLOBAL_V, st["global_v"])
        dsm_set_round(self.h, st["round"])
        dsm_set_gamma(self.h, st["gamma"])

    def close(self):
        if getattr(self, "h", None) is not None:
            dsm_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
