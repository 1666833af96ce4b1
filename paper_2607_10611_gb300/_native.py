"""ctypes binding of the C ABI in include/mpadam.h (argument marshalling only).

Every function here has the name of the C entry point it calls, takes device
pointers as Python ints, raises MPAdamError carrying mpadam_last_error() on
a non-OK status, and does no computation of its own.  The library must have
been built (paper_2607_10611_gb300.build()); there is no fallback.
"""
from __future__ import annotations

import ctypes
import math
from typing import Optional, Sequence

from . import builder as _build

MPADAM_OK, MPADAM_EINVAL, MPADAM_EALLOC, MPADAM_ECUDA, MPADAM_EUNSUPPORTED = 0, 1, 2, 3, 4
MPADAM_F32, MPADAM_BF16, MPADAM_E4M3, MPADAM_E4M3_B32, MPADAM_NVFP4 = 0, 1, 2, 3, 4
MPADAM_ROUND_NEAREST, MPADAM_ROUND_STOCHASTIC = 0, 1
DTYPE = {"f32": MPADAM_F32, "bf16": MPADAM_BF16, "e4m3": MPADAM_E4M3, "e4m3_b32": MPADAM_E4M3_B32,
         "nvfp4": MPADAM_NVFP4}
ROUNDING = {"nearest": MPADAM_ROUND_NEAREST, "stochastic": MPADAM_ROUND_STOCHASTIC}

EXPORTED = ["mpadam_create", "mpadam_create_ex", "mpadam_fp8_init", "mpadam_step", "mpadam_step_host",
            "mpadam_destroy", "mpadam_last_error", "mpadam_global_offset", "mpadam_global_length", "mpadam_set_grid",
            "mpadam_set_tail_pool", "mpadam_launch_info", "mpadam_rng_lanes", "mpadam_step_noalloc", "mpadam_noalloc_status", "mpadam_device_status",
            "mpadam_toy_create", "mpadam_toy_step", "mpadam_toy_run", "mpadam_toy_destroy", "mpadam_host_buffer_alloc",
            "mpadam_host_buffer_free", "mpadam_debug_fail_allocation", "mpadam_debug_tile_schedule"]


class MPAdamError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"mpadam status {status}: {message}")
        self.status = status


class mpadam_tensor(ctypes.Structure):
    _fields_ = [("w", ctypes.c_void_p), ("m", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("ve", ctypes.c_void_p), ("numel", ctypes.c_int64)]


class mpadam_tensor_ex(ctypes.Structure):
    _fields_ = [("w", ctypes.c_void_p), ("m", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("ve", ctypes.c_void_p), ("numel", ctypes.c_int64), ("weight_dtype", ctypes.c_int32),
                ("global_scale", ctypes.c_float), ("block_scale", ctypes.c_void_p), ("compute", ctypes.c_void_p)]


class mpadam_config(ctypes.Structure):
    _fields_ = [
        ("lr_add", ctypes.c_float), ("lr_mul", ctypes.c_float),
        ("beta1", ctypes.c_float), ("beta2", ctypes.c_float),
        ("eps", ctypes.c_float), ("tau", ctypes.c_float),
        ("rmax_pos", ctypes.c_float), ("rmax_neg", ctypes.c_float),
        ("g_max", ctypes.c_float), ("dmult_max", ctypes.c_float),
        ("w_max", ctypes.c_float), ("wd_add", ctypes.c_float),
        ("bias_correction", ctypes.c_int32), ("rounding", ctypes.c_int32),
        ("seed", ctypes.c_uint64),
        ("weight_dtype", ctypes.c_int32), ("grad_dtype", ctypes.c_int32),
        ("moment_dtype", ctypes.c_int32), ("reserved", ctypes.c_int32),
    ]


class mpadam_toy_config(ctypes.Structure):
    _fields_ = [("mode", ctypes.c_int32), ("split", ctypes.c_int32), ("batch", ctypes.c_int32),
                ("reserved", ctypes.c_int32), ("lr_add", ctypes.c_float), ("lr_mul", ctypes.c_float),
                ("rmax", ctypes.c_float), ("tau", ctypes.c_float), ("c_lo", ctypes.c_float),
                ("c_hi", ctypes.c_float), ("seed", ctypes.c_uint64)]


TOY_MODES = {"additive": 0, "multiplicative": 1, "combined": 2}


CONFIG_DEFAULTS = dict(lr_add=1e-3, lr_mul=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, tau=1e-8,
                       rmax_pos=0.75, rmax_neg=0.75, g_max=math.inf, dmult_max=math.inf,
                       w_max=math.inf, wd_add=0.0, bias_correction=1, rounding=MPADAM_ROUND_NEAREST,
                       seed=0, weight_dtype=MPADAM_BF16, grad_dtype=MPADAM_F32,
                       moment_dtype=MPADAM_F32, reserved=0)


def make_config(**kw) -> mpadam_config:
    d = dict(CONFIG_DEFAULTS)
    for k, v in kw.items():
        if k not in d:
            raise KeyError(k)
        if k in ("weight_dtype", "grad_dtype", "moment_dtype") and isinstance(v, str):
            v = DTYPE[v]
        if k == "rounding" and isinstance(v, str):
            v = ROUNDING[v]
        d[k] = v
    return mpadam_config(**d)


_LIB: Optional[ctypes.CDLL] = None


def lib() -> ctypes.CDLL:
    global _LIB
    if _LIB is None:
        if not _build.LIB.exists():
            raise RuntimeError(f"{_build.LIB} is missing: build the CUDA library first "
                               "(paper_2607_10611_gb300.build())")
        L = ctypes.CDLL(str(_build.LIB))
        P, i32, i64, u64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64
        sig = {
            "mpadam_create": [P, i32, P, P, P, P],
            "mpadam_create_ex": [P, i32, P, P, P, P],
            "mpadam_fp8_init": [P, P, i64, P],
            "mpadam_step": [P, P, i64, P],
            "mpadam_step_host": [P, P, P, i64, P],
            "mpadam_destroy": [P],
            "mpadam_global_offset": [P, i32, P],
            "mpadam_global_length": [P, P],
            "mpadam_set_grid": [P, i32],
            "mpadam_set_tail_pool": [P, i32, i32],
            "mpadam_launch_info": [P, P, P],
            "mpadam_rng_lanes": [u64, i64, i32, i64, i64, P, P],
            "mpadam_step_noalloc": [P, i32, P, P, P, P, i64, P],
            "mpadam_device_status": [P, P],
            "mpadam_noalloc_status": [P, P],
            "mpadam_toy_create": [i64, P, P],
            "mpadam_toy_step": [P, P, P, i64, P, P],
            "mpadam_toy_run": [P, P, P, i64, i64, P, P],
            "mpadam_toy_destroy": [P],
            "mpadam_host_buffer_alloc": [i64, P],
            "mpadam_host_buffer_free": [P, i64],
            "mpadam_debug_fail_allocation": [i32],
            "mpadam_debug_tile_schedule": [P, i32, i32, i32, i32, P, P, P, i32, P],
        }
        for name, args in sig.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = i32
        L.mpadam_last_error.argtypes = []
        L.mpadam_last_error.restype = ctypes.c_char_p
        _LIB = L
    return _LIB


def mpadam_last_error() -> str:
    return lib().mpadam_last_error().decode(errors="replace")


def _check(status: int) -> None:
    if status != MPADAM_OK:
        raise MPAdamError(status, mpadam_last_error())


def _ptr_array(ptrs: Sequence[int]):
    arr = (ctypes.c_void_p * max(1, len(ptrs)))()
    for i, p in enumerate(ptrs):
        arr[i] = p
    return arr


def mpadam_create(tensors: Sequence[tuple], cfg: mpadam_config, fp8_exp: int = 0, fp8_amax: int = 0) -> int:
    """tensors: (w, m, v, ve, numel) per tensor, pointers as ints.  Returns the state handle."""
    arr = (mpadam_tensor * max(1, len(tensors)))()
    for i, (w, m, v, ve, n) in enumerate(tensors):
        arr[i] = mpadam_tensor(w, m, v, ve, n)
    out = ctypes.c_void_p()
    _check(lib().mpadam_create(arr, len(tensors), ctypes.byref(cfg), fp8_exp or None, fp8_amax or None,
                               ctypes.byref(out)))
    return out.value


def mpadam_create_ex(tensors: Sequence[tuple], cfg: mpadam_config, fp8_exp: int = 0, fp8_amax: int = 0) -> int:
    """tensors: (w, m, v, ve, numel, weight_dtype, block_scale, compute[, global_scale]) per
    tensor, pointers as ints (0 = NULL), weight_dtype an MPADAM_* value or its name,
    global_scale the NVFP4 tensor scale (0 for other formats)."""
    arr = (mpadam_tensor_ex * max(1, len(tensors)))()
    for i, t in enumerate(tensors):
        w, m, v, ve, n, wd, bs, cc = t[:8]
        gs = float(t[8]) if len(t) > 8 else 0.0
        arr[i] = mpadam_tensor_ex(w, m, v, ve, n, DTYPE[wd] if isinstance(wd, str) else wd, gs, bs or None,
                                  cc or None)
    out = ctypes.c_void_p()
    _check(lib().mpadam_create_ex(arr, len(tensors), ctypes.byref(cfg), fp8_exp or None, fp8_amax or None,
                                  ctypes.byref(out)))
    return out.value


def mpadam_fp8_init(state: int, init_exp: Sequence[int], first_step: int, stream: int = 0) -> None:
    arr = (ctypes.c_int32 * max(1, len(init_exp)))(*init_exp)
    _check(lib().mpadam_fp8_init(state, arr, first_step, stream or None))


def mpadam_step(state: int, grads: Sequence[int], step: int, stream: int = 0) -> None:
    _check(lib().mpadam_step(state, _ptr_array(grads), step, stream or None))


def mpadam_step_host(state: int, host_grads: Sequence[int], host_w_out: Sequence[int], step: int,
                     stream: int = 0) -> None:
    _check(lib().mpadam_step_host(state, _ptr_array(host_grads), _ptr_array(host_w_out), step,
                                  stream or None))


def mpadam_destroy(state: int) -> None:
    _check(lib().mpadam_destroy(state))


def mpadam_global_offset(state: int, k: int) -> int:
    out = ctypes.c_int64()
    _check(lib().mpadam_global_offset(state, k, ctypes.byref(out)))
    return out.value


def mpadam_global_length(state: int) -> int:
    out = ctypes.c_int64()
    _check(lib().mpadam_global_length(state, ctypes.byref(out)))
    return out.value


def mpadam_set_grid(state: int, ctas: int) -> None:
    _check(lib().mpadam_set_grid(state, ctas))


def mpadam_set_tail_pool(state: int, static_q: int, chunk_tiles: int) -> None:
    _check(lib().mpadam_set_tail_pool(state, static_q, chunk_tiles))


def mpadam_launch_info(state: int) -> tuple:
    c, t = ctypes.c_int32(), ctypes.c_int32()
    _check(lib().mpadam_launch_info(state, ctypes.byref(c), ctypes.byref(t)))
    return c.value, t.value


def mpadam_device_status(state: int) -> int:
    """Synchronises; returns and clears the step kernel's device error bits."""
    out = ctypes.c_int32()
    _check(lib().mpadam_device_status(state, ctypes.byref(out)))
    return out.value


def mpadam_rng_lanes(seed: int, step: int, weight_dtype: int, first: int, n: int, out: int,
                     stream: int = 0) -> None:
    _check(lib().mpadam_rng_lanes(seed, step, weight_dtype, first, n, out, stream or None))


def mpadam_step_noalloc(tensors: Sequence[tuple], grads: Sequence[int], cfg: mpadam_config, step: int,
                        fp8_exp: int = 0, fp8_amax: int = 0, stream: int = 0) -> None:
    """Allocation-free step: tensors as for mpadam_create, grads as for mpadam_step."""
    arr = (mpadam_tensor * max(1, len(tensors)))()
    for i, (w, m, v, ve, n) in enumerate(tensors):
        arr[i] = mpadam_tensor(w, m, v, ve, n)
    _check(lib().mpadam_step_noalloc(arr, len(tensors), _ptr_array(grads), ctypes.byref(cfg),
                                     fp8_exp or None, fp8_amax or None, step, stream or None))


def mpadam_noalloc_status(stream: int = 0) -> int:
    """Waits for `stream`; returns and clears the allocation-free steps'
    device error bits (0: no bounded wait gave up)."""
    out = ctypes.c_int32()
    _check(lib().mpadam_noalloc_status(stream or None, ctypes.byref(out)))
    return out.value


def mpadam_toy_create(n: int, cfg: mpadam_toy_config) -> int:
    out = ctypes.c_void_p()
    _check(lib().mpadam_toy_create(n, ctypes.byref(cfg), ctypes.byref(out)))
    return out.value


def mpadam_toy_step(state: int, w: int, wstar: int, step: int, loss_out: int = 0, stream: int = 0) -> None:
    _check(lib().mpadam_toy_step(state, w, wstar, step, loss_out or None, stream or None))


def mpadam_toy_run(state: int, w: int, wstar: int, first_step: int, steps: int, losses: int = 0,
                   stream: int = 0) -> None:
    _check(lib().mpadam_toy_run(state, w, wstar, first_step, steps, losses or None, stream or None))


def mpadam_toy_destroy(state: int) -> None:
    _check(lib().mpadam_toy_destroy(state))


def mpadam_host_buffer_alloc(nbytes: int) -> int:
    out = ctypes.c_void_p()
    _check(lib().mpadam_host_buffer_alloc(nbytes, ctypes.byref(out)))
    return out.value


def mpadam_host_buffer_free(ptr: int, nbytes: int) -> None:
    _check(lib().mpadam_host_buffer_free(ptr, nbytes))


def mpadam_debug_fail_allocation(after: int) -> None:
    """Test hook: the library's allocation after `after` more successful ones
    fails once (-1 disarms)."""
    _check(lib().mpadam_debug_fail_allocation(after))


def mpadam_debug_tile_schedule(numel, ctas: int, static_q: int, chunk_tiles: int):
    """The step's tile schedule, computed on the host: per CTA (tb, ts, te)
    and its first tensor, and the tail pool's chunks (start, count, tensor)."""
    import numpy as np
    nm = np.ascontiguousarray(numel, dtype=np.int64)
    runs = np.zeros((ctas, 3), dtype=np.int64)
    first = np.zeros(ctas, dtype=np.int32)
    count = ctypes.c_int32(0)
    cap = 0
    while True:
        pool = np.zeros((max(cap, 1), 3), dtype=np.int64)
        rc = lib().mpadam_debug_tile_schedule(nm.ctypes.data, len(nm), ctas, static_q, chunk_tiles,
                                               runs.ctypes.data, first.ctypes.data, pool.ctypes.data, cap,
                                               ctypes.byref(count))
        if rc == MPADAM_EINVAL and count.value > cap:
            cap = count.value
            continue
        _check(rc)
        return runs, first, pool[:count.value]
