"""Python binding of the kvdro C ABI (include/kvdro.h).

Argument marshalling only: every function here converts its arguments to plain
pointers and sizes and calls the entry point of the same name in
``_build/libkvdro.so``.  Every step of the computation runs in that library's
CUDA kernels; there is no CPU or PyTorch path.  If the library is missing or
cannot be loaded, the first call raises.

Array arguments may be NumPy arrays (host memory) or torch tensors (host or
CUDA memory); the library itself tells host from device pointers.  Streams may
be a ``torch.cuda.Stream``, a raw ``cudaStream_t`` integer, or None (the legacy
default stream).
"""

from __future__ import annotations

import ctypes
import os
import threading
from typing import Any

import numpy as np

from . import build as _build

KVDRO_OK = 0
KVDRO_EINVAL = -1
KVDRO_ENOMEM = -2
KVDRO_ECUDA = -3
KVDRO_ESTATE = -4
KVDRO_ETIMEOUT = -5
KVDRO_FP32 = 0
KVDRO_FP64 = 1
KVDRO_EXACT = 2
KVDRO_ENVELOPE = 3

_STATUS = {0: "KVDRO_OK", -1: "KVDRO_EINVAL", -2: "KVDRO_ENOMEM", -3: "KVDRO_ECUDA", -4: "KVDRO_ESTATE",
           -5: "KVDRO_ETIMEOUT"}

# Every entry point declared in include/kvdro.h.
SYMBOLS = ("kvdro_create", "kvdro_load_samples", "kvdro_quantiles", "kvdro_eval_grid", "kvdro_sorted_samples",
           "kvdro_eval_dual", "kvdro_last_grid_ms", "kvdro_eval_grid_noalloc", "kvdro_sync", "kvdro_last_error", "kvdro_destroy")

_lock = threading.Lock()
_lib = None


class KvdroError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{_STATUS.get(status, status)}: {message}")
        self.status = status


def library_path() -> str:
    return _build.LIB


def load_library(build_if_missing: bool = True) -> ctypes.CDLL:
    """Load libkvdro.so (building it with nvcc first if it is absent)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = _build.LIB
        if not os.path.exists(path):
            if not build_if_missing:
                raise RuntimeError(f"kvdro CUDA library not built: {path}")
            _build.build()
        lib = ctypes.CDLL(path)
        P, i32 = ctypes.c_void_p, ctypes.c_int32
        lib.kvdro_create.restype = ctypes.c_int
        lib.kvdro_create.argtypes = [ctypes.POINTER(P), ctypes.c_int]
        lib.kvdro_load_samples.restype = ctypes.c_int
        lib.kvdro_load_samples.argtypes = [P, i32, P, P, P, P, P]
        lib.kvdro_quantiles.restype = ctypes.c_int
        lib.kvdro_quantiles.argtypes = [P, i32, P, P, P]
        lib.kvdro_eval_grid.restype = ctypes.c_int
        lib.kvdro_eval_grid.argtypes = [P, ctypes.c_int, i32, P, i32, P, i32, P, i32, P, P, P, P, P, P, P, P, P]
        lib.kvdro_eval_dual.restype = ctypes.c_int
        lib.kvdro_eval_dual.argtypes = [P, i32, P, i32, P, i32, P, P, P, P, P, P, P, P]
        lib.kvdro_sorted_samples.restype = ctypes.c_int
        lib.kvdro_sorted_samples.argtypes = [P, P, P]
        lib.kvdro_last_grid_ms.restype = ctypes.c_int
        lib.kvdro_last_grid_ms.argtypes = [P, ctypes.POINTER(ctypes.c_float)]
        lib.kvdro_eval_grid_noalloc.restype = ctypes.c_int
        lib.kvdro_eval_grid_noalloc.argtypes = [i32, P, P, P, P, i32, P, i32, P, i32, P, i32, P, P, P, P, P, P, P, P,
                                                ctypes.c_char_p, i32]
        lib.kvdro_sync.restype = ctypes.c_int
        lib.kvdro_sync.argtypes = [P]
        lib.kvdro_last_error.restype = ctypes.c_char_p
        lib.kvdro_last_error.argtypes = [P]
        lib.kvdro_destroy.restype = ctypes.c_int
        lib.kvdro_destroy.argtypes = [P]
        _lib = lib
        return lib


# ------------------------------------------------------------------ marshalling

def _ptr(a: Any, dtype=None):
    """Pointer to the data of a NumPy array or torch tensor (None -> NULL)."""
    if a is None:
        return None
    if isinstance(a, np.ndarray):
        if dtype is not None and a.dtype != np.dtype(dtype):
            raise TypeError(f"expected dtype {np.dtype(dtype)}, got {a.dtype}")
        if not a.flags["C_CONTIGUOUS"]:
            raise ValueError("array must be C-contiguous")
        return a.ctypes.data
    if hasattr(a, "data_ptr"):
        if dtype is not None:
            want = np.dtype(dtype).name
            got = str(a.dtype).replace("torch.", "")
            if got != want:
                raise TypeError(f"expected dtype {want}, got {got}")
        if not a.is_contiguous():
            raise ValueError("tensor must be contiguous")
        return a.data_ptr()
    raise TypeError(f"unsupported array type {type(a)}")


def _host(a: Any, dtype) -> np.ndarray:
    """Small host-side parameter arrays are converted to contiguous NumPy of the ABI dtype."""
    if hasattr(a, "detach"):
        a = a.detach().cpu().numpy()
    return np.ascontiguousarray(np.asarray(a), dtype=dtype)


def _stream(s: Any):
    if s is None:
        return None
    if isinstance(s, int):
        return s
    if hasattr(s, "cuda_stream"):
        return s.cuda_stream
    raise TypeError(f"unsupported stream {type(s)}")


def _numel(a: Any) -> int:
    if isinstance(a, np.ndarray):
        return int(a.size)
    if hasattr(a, "numel"):
        return int(a.numel())
    return int(np.asarray(a).size)


def _need(name: str, a: Any, n: int) -> None:
    """Raise ValueError unless array ``a`` (if given) holds exactly ``n`` elements: the library
    reads or writes exactly that many through the pointer, so a shorter buffer would be
    overrun (on the device or on the host)."""
    if a is not None and _numel(a) != n:
        raise ValueError(f"{name} has {_numel(a)} elements; the call needs exactly {n}")


def _on_device(name: str, a: Any) -> None:
    if a is not None and not (hasattr(a, "is_cuda") and a.is_cuda):
        raise ValueError(f"{name} must be a CUDA tensor")


# Class count and sample total of each context's loaded samples (keyed by the handle), so
# that outputs sized by them can be checked before a call.
_loaded: dict = {}


def _check(ctx, status: int):
    if status != KVDRO_OK:
        msg = load_library().kvdro_last_error(ctx).decode() if ctx else ""
        raise KvdroError(status, msg)


# ------------------------------------------------------------------ entry points

def kvdro_create(device_ordinal: int = 0) -> ctypes.c_void_p:
    lib = load_library()
    h = ctypes.c_void_p()
    st = lib.kvdro_create(ctypes.byref(h), int(device_ordinal))
    if st != KVDRO_OK:
        raise KvdroError(st, f"kvdro_create(device={device_ordinal}) failed")
    return h


def _check_samples(K: int, off: np.ndarray, lengths, lm: np.ndarray, li) -> None:
    if int(K) < 1:
        raise ValueError(f"K = {K} must be at least 1")
    _need("offsets", off, int(K) + 1)
    _need("L_max", lm, int(K))
    _need("L_in", li, int(K))
    _need("lengths", lengths, int(off[-1]))


def kvdro_load_samples(ctx, K: int, offsets, lengths, L_max, L_in=None, stream=None) -> None:
    off = _host(offsets, np.int64)
    lm = _host(L_max, np.int32)
    li = None if L_in is None else _host(L_in, np.int32)
    _check_samples(K, off, lengths, lm, li)
    key = getattr(ctx, "value", ctx)
    _loaded.pop(key, None)
    _check(ctx, load_library().kvdro_load_samples(ctx, int(K), off.ctypes.data, _ptr(lengths, np.int32), lm.ctypes.data,
                                                  None if li is None else li.ctypes.data, _stream(stream)))
    _loaded[key] = (int(K), int(off[-1]))


def _ctx_K(ctx):
    """Class count of the context's loaded samples (None if unknown here)."""
    got = _loaded.get(getattr(ctx, "value", ctx))
    return None if got is None else got[0]


def kvdro_quantiles(ctx, F: int, fractiles, out, stream=None) -> None:
    fr = _host(fractiles, np.float64)
    _need("fractiles", fr, int(F))
    K = _ctx_K(ctx)
    if K is not None:
        _need("out", out, K * int(F))
    _check(ctx, load_library().kvdro_quantiles(ctx, int(F), fr.ctypes.data, _ptr(out, np.int32), _stream(stream)))


def _check_grid(R, rr, E, ee, M, cp, cw, NL=None, ll=None) -> None:
    _need("r", rr, int(R))
    if NL is not None:
        _need("lam", ll, int(NL))
    _need("eps", ee, int(E))
    _need("c_p", cp, int(M))
    _need("c_w", cw, int(M))


def _check_outputs(K: int, R: int, E: int, M: int, NL=None, **outs) -> None:
    rows = M * E * K
    size = {"S": M * K * R * (NL or 0), "cost": rows * R, "lam_idx": rows * R, "gamma": rows * R, "r_idx": rows,
            "min_cost": rows, "fhat": rows}
    for name, a in outs.items():
        _need(name, a, size[name])


def kvdro_eval_grid(ctx, precision: int, R: int, r, NL: int, lam, E: int, eps, M: int, c_p, c_w, S=None, cost=None,
                    lam_idx=None, r_idx=None, min_cost=None, fhat=None, stream=None) -> None:
    ft = np.float32 if precision == KVDRO_FP32 else np.float64
    rr, ll, ee = _host(r, np.int32), _host(lam, np.float64), _host(eps, np.float64)
    cp, cw = _host(c_p, np.float64), _host(c_w, np.float64)
    _check_grid(R, rr, E, ee, M, cp, cw, NL=NL, ll=ll)
    K = _ctx_K(ctx)
    if K is not None:
        _check_outputs(K, int(R), int(E), int(M), NL=int(NL), S=S, cost=cost, lam_idx=lam_idx, r_idx=r_idx,
                       min_cost=min_cost, fhat=fhat)
    _check(ctx, load_library().kvdro_eval_grid(
        ctx, int(precision), int(R), rr.ctypes.data, int(NL), ll.ctypes.data, int(E), ee.ctypes.data, int(M),
        cp.ctypes.data, cw.ctypes.data, _ptr(S, ft), _ptr(cost, ft), _ptr(lam_idx, np.int32), _ptr(r_idx, np.int32),
        _ptr(min_cost, ft), _ptr(fhat, np.float64), _stream(stream)))


def kvdro_eval_dual(ctx, R: int, r, E: int, eps, M: int, c_p, c_w, cost=None, gamma=None, r_idx=None,
                    min_cost=None, fhat=None, stream=None) -> None:
    rr, ee = _host(r, np.int32), _host(eps, np.float64)
    cp, cw = _host(c_p, np.float64), _host(c_w, np.float64)
    _check_grid(R, rr, E, ee, M, cp, cw)
    K = _ctx_K(ctx)
    if K is not None:
        _check_outputs(K, int(R), int(E), int(M), cost=cost, gamma=gamma, r_idx=r_idx, min_cost=min_cost, fhat=fhat)
    _check(ctx, load_library().kvdro_eval_dual(
        ctx, int(R), rr.ctypes.data, int(E), ee.ctypes.data, int(M), cp.ctypes.data, cw.ctypes.data,
        _ptr(cost, np.float64), _ptr(gamma, np.float64), _ptr(r_idx, np.int32), _ptr(min_cost, np.float64),
        _ptr(fhat, np.float64), _stream(stream)))


def kvdro_sorted_samples(ctx, out, stream=None) -> None:
    got = _loaded.get(getattr(ctx, "value", ctx))
    if got is not None:
        _need("out", out, got[1])
    _check(ctx, load_library().kvdro_sorted_samples(ctx, _ptr(out, np.int32), _stream(stream)))


def kvdro_last_grid_ms(ctx) -> float:
    ms = ctypes.c_float()
    _check(ctx, load_library().kvdro_last_grid_ms(ctx, ctypes.byref(ms)))
    return float(ms.value)


def kvdro_eval_grid_noalloc(K: int, offsets, lengths, L_max, L_in, R: int, r, NL: int, lam, E: int, eps, M: int,
                            c_p, c_w, cost=None, lam_idx=None, r_idx=None, min_cost=None, fhat=None,
                            stream=None) -> None:
    """FP32 grid pass in the library's static scratch (allocates nothing; see include/kvdro.h).
    ``lengths`` and the outputs must be CUDA tensors on the current device."""
    off, lm = _host(offsets, np.int64), _host(L_max, np.int32)
    li = None if L_in is None else _host(L_in, np.int32)
    rr, ll, ee = _host(r, np.int32), _host(lam, np.float64), _host(eps, np.float64)
    cp, cw = _host(c_p, np.float64), _host(c_w, np.float64)
    _check_samples(K, off, lengths, lm, li)
    _check_grid(R, rr, E, ee, M, cp, cw, NL=NL, ll=ll)
    _check_outputs(int(K), int(R), int(E), int(M), cost=cost, lam_idx=lam_idx, r_idx=r_idx, min_cost=min_cost,
                   fhat=fhat)
    for name, a in (("lengths", lengths), ("cost", cost), ("lam_idx", lam_idx), ("r_idx", r_idx),
                    ("min_cost", min_cost), ("fhat", fhat)):
        _on_device(name, a)
    buf = ctypes.create_string_buffer(512)
    st = load_library().kvdro_eval_grid_noalloc(
        int(K), off.ctypes.data, _ptr(lengths, np.int32), lm.ctypes.data, None if li is None else li.ctypes.data,
        int(R), rr.ctypes.data, int(NL), ll.ctypes.data, int(E), ee.ctypes.data, int(M), cp.ctypes.data,
        cw.ctypes.data, _ptr(cost, np.float32), _ptr(lam_idx, np.int32), _ptr(r_idx, np.int32),
        _ptr(min_cost, np.float32), _ptr(fhat, np.float64), _stream(stream), buf, len(buf))
    if st != KVDRO_OK:
        raise KvdroError(st, buf.value.decode())


def kvdro_sync(ctx) -> None:
    _check(ctx, load_library().kvdro_sync(ctx))


def kvdro_last_error(ctx) -> str:
    return load_library().kvdro_last_error(ctx).decode()


def kvdro_destroy(ctx) -> None:
    if ctx:
        _loaded.pop(getattr(ctx, "value", ctx), None)
        load_library().kvdro_destroy(ctx)
