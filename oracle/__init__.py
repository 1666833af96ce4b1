"""CPU oracle of the M+Adam optimizer step (arxiv 2607.10611) -- ctypes wrapper.

TEST INFRASTRUCTURE ONLY.  The oracle is a plain, single-threaded C
implementation (mpadam_oracle.c) of Algorithm 1 with the options of
Algorithm 2 (Appendix A), in IEEE binary32 as the paper's FP32-compute /
low-precision-storage round trip prescribes (Appendix B).  Only the tests, the
smoke check and the benchmark's CPU-baseline leg may import this package; the
CUDA library never does, and this package imports nothing from it.

Arrays are numpy: float32 for FP32, uint16 bit patterns for BF16, uint8 codes
for E4M3.  Functions update their arguments in place where stated.
"""
from __future__ import annotations

import ctypes
import math
from typing import List, Optional, Sequence

import numpy as np

from . import build as _build

F32, BF16, E4M3, E4M3_B32, NVFP4 = 0, 1, 2, 3, 4
DTYPES = {"f32": F32, "bf16": BF16, "e4m3": E4M3, "e4m3_b32": E4M3_B32, "nvfp4": NVFP4}
ALIGN = 8
BLOCK = 32
FP4_BLOCK = 16

_LIB = None


class HParams(ctypes.Structure):
    _fields_ = [
        ("lr_add", ctypes.c_float), ("lr_mul", ctypes.c_float),
        ("beta1", ctypes.c_float), ("beta2", ctypes.c_float),
        ("eps", ctypes.c_float), ("tau", ctypes.c_float),
        ("rmax_pos", ctypes.c_float), ("rmax_neg", ctypes.c_float),
        ("g_max", ctypes.c_float), ("dmult_max", ctypes.c_float),
        ("w_max", ctypes.c_float), ("wd_add", ctypes.c_float),
        ("bias_correction", ctypes.c_int32), ("stochastic", ctypes.c_int32),
        ("seed", ctypes.c_uint64),
    ]


class Scalars(ctypes.Structure):
    _fields_ = [(n, ctypes.c_float) for n in
                ("b1", "b2", "omb1", "omb2", "ka", "c2", "km", "ln2", "eps", "tau",
                 "lo", "hi", "gmax", "wmax", "kwd")] + \
               [("gmax_on", ctypes.c_int32), ("wmax_on", ctypes.c_int32), ("wd_on", ctypes.c_int32)]


DEFAULTS = dict(lr_add=1e-3, lr_mul=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, tau=1e-8,
                rmax_pos=0.75, rmax_neg=0.75, g_max=math.inf, dmult_max=math.inf,
                w_max=math.inf, wd_add=0.0, bias_correction=1, stochastic=0, seed=0)


def hparams(**kw) -> HParams:
    d = dict(DEFAULTS)
    for k, val in kw.items():
        if k not in d:
            raise KeyError(k)
        d[k] = val
    return HParams(**d)


def lib() -> ctypes.CDLL:
    global _LIB
    if _LIB is None:
        path = _build.build()
        L = ctypes.CDLL(str(path))
        P, i64, i32, u64 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_uint64
        L.orc_philox4x32_10.argtypes = [P, P, P]
        L.orc_rng_lane.argtypes = [u64, u64, u64, i32]
        L.orc_rng_lane.restype = ctypes.c_uint32
        L.orc_bf16_rne.argtypes = [ctypes.c_float]; L.orc_bf16_rne.restype = ctypes.c_uint16
        L.orc_bf16_sr.argtypes = [ctypes.c_float, ctypes.c_uint32]; L.orc_bf16_sr.restype = ctypes.c_uint16
        L.orc_e4m3_rne.argtypes = [ctypes.c_float]; L.orc_e4m3_rne.restype = ctypes.c_uint8
        L.orc_e4m3_sr.argtypes = [ctypes.c_float, ctypes.c_uint32]; L.orc_e4m3_sr.restype = ctypes.c_uint8
        L.orc_e4m3_decode.argtypes = [ctypes.c_uint8]; L.orc_e4m3_decode.restype = ctypes.c_float
        L.orc_fp8_next_exponent.argtypes = [ctypes.c_float, i32]; L.orc_fp8_next_exponent.restype = i32
        L.orc_scalars_for_step.argtypes = [P, i64, P]; L.orc_scalars_for_step.restype = i32
        L.orc_step_elements.argtypes = [i64, P, i64, i32, i32, i32, P, P, P, P, P, P, i64, i32, i32, P]
        L.orc_step_elements.restype = i32
        L.orc_e4m3_amax.argtypes = [i64, P, i32]; L.orc_e4m3_amax.restype = ctypes.c_float
        L.orc_bf16_rne_n.argtypes = [i64, P, P]
        L.orc_bf16_sr_n.argtypes = [i64, P, P, P]
        L.orc_e4m3_rne_n.argtypes = [i64, P, P]
        L.orc_e4m3_sr_n.argtypes = [i64, P, P, P]
        L.orc_e4m3_decode_n.argtypes = [i64, P, P]
        L.orc_rng_lanes_n.argtypes = [u64, u64, i32, i64, P, P]
        L.orc_philox_n.argtypes = [i64, P, P, P]
        L.orc_update_elements_n.argtypes = [P, i64, i64, P, P, P, P, P, P, P, P, P]
        L.orc_update_elements_n.restype = i32
        L.orc_fp16_pow2.argtypes = [i32]; L.orc_fp16_pow2.restype = ctypes.c_uint16
        L.orc_fp16_decode.argtypes = [ctypes.c_uint16]; L.orc_fp16_decode.restype = ctypes.c_float
        L.orc_block_exponent.argtypes = [ctypes.c_float, i32]; L.orc_block_exponent.restype = i32
        L.orc_step_block_e4m3.argtypes = [i64, i64, i32, i32, P, P, P, P, P, P, P, i64]
        L.orc_step_block_e4m3.restype = i32
        L.orc_dequant_bf16.argtypes = [i64, P, i32, P, P]
        L.orc_e2m1_rne.argtypes = [ctypes.c_float]; L.orc_e2m1_rne.restype = ctypes.c_uint8
        L.orc_e2m1_sr.argtypes = [ctypes.c_float, ctypes.c_uint32]; L.orc_e2m1_sr.restype = ctypes.c_uint8
        L.orc_e2m1_decode.argtypes = [ctypes.c_uint8]; L.orc_e2m1_decode.restype = ctypes.c_float
        L.orc_nvfp4_scale_code.argtypes = [ctypes.c_float, ctypes.c_float, i32]
        L.orc_nvfp4_scale_code.restype = i32
        L.orc_step_nvfp4.argtypes = [i64, i64, i32, i32, P, P, ctypes.c_float, P, P, P, P, P, i64]
        L.orc_step_nvfp4.restype = i32
        L.orc_dequant_nvfp4_bf16.argtypes = [i64, P, P, ctypes.c_float, P]
        L.orc_tree_sum.argtypes = [i64, P]; L.orc_tree_sum.restype = ctypes.c_double
        L.orc_toy_step.argtypes = [P, i64, P, P, i64]; L.orc_toy_step.restype = ctypes.c_double
        _LIB = L
    return _LIB


def _p(a: np.ndarray):
    return ctypes.c_void_p(a.ctypes.data)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


# --------------------------------------------------------------------------
# Random bits
# --------------------------------------------------------------------------
def philox4x32_10(ctr: Sequence[int], key: Sequence[int]) -> np.ndarray:
    c = _c(ctr, np.uint32).reshape(-1)
    k = _c(key, np.uint32)
    out = np.zeros(c.size, np.uint32)
    lib().orc_philox_n(c.size // 4, _p(c), _p(k), _p(out))
    return out


def rng_lanes(seed: int, t: int, idx, storage: int) -> np.ndarray:
    """Random bits the step draws for global element indices `idx` at step t:
    16-bit lanes for BF16 storage, 32-bit lanes for E4M3 storage."""
    i = _c(idx, np.uint64)
    out = np.zeros(i.size, np.uint32)
    lib().orc_rng_lanes_n(seed, t, storage, i.size, _p(i), _p(out))
    return out


# --------------------------------------------------------------------------
# Storage formats
# --------------------------------------------------------------------------
def bf16_rne(x) -> np.ndarray:
    x = _c(x, np.float32); out = np.zeros(x.size, np.uint16)
    lib().orc_bf16_rne_n(x.size, _p(x), _p(out)); return out


def bf16_sr(x, r16) -> np.ndarray:
    x = _c(x, np.float32); r = _c(r16, np.uint32); out = np.zeros(x.size, np.uint16)
    lib().orc_bf16_sr_n(x.size, _p(x), _p(r), _p(out)); return out


def bf16_decode(h) -> np.ndarray:
    return (_c(h, np.uint16).astype(np.uint32) << 16).view(np.float32)


def e4m3_rne(x) -> np.ndarray:
    x = _c(x, np.float32); out = np.zeros(x.size, np.uint8)
    lib().orc_e4m3_rne_n(x.size, _p(x), _p(out)); return out


def e4m3_sr(x, r32) -> np.ndarray:
    x = _c(x, np.float32); r = _c(r32, np.uint32); out = np.zeros(x.size, np.uint8)
    lib().orc_e4m3_sr_n(x.size, _p(x), _p(r), _p(out)); return out


def e4m3_decode(q) -> np.ndarray:
    q = _c(q, np.uint8); out = np.zeros(q.size, np.float32)
    lib().orc_e4m3_decode_n(q.size, _p(q), _p(out)); return out


def fp8_next_exponent(amax: float, e_cur: int) -> int:
    return int(lib().orc_fp8_next_exponent(ctypes.c_float(amax), int(e_cur)))


def e4m3_amax(q, e: int) -> float:
    q = _c(q, np.uint8)
    return float(lib().orc_e4m3_amax(q.size, _p(q), int(e)))


# --------------------------------------------------------------------------
# The update
# --------------------------------------------------------------------------
def scalars(hp: HParams, t: int) -> Scalars:
    s = Scalars()
    if lib().orc_scalars_for_step(ctypes.byref(hp), t, ctypes.byref(s)) != 0:
        raise ValueError("invalid hyper-parameters or step")
    return s


def update_elements(hp: HParams, t: int, w, g, m, v, ve):
    """The binary32 update without storage rounding: returns (wn, m1, v1, ve1)."""
    arrs = [_c(a, np.float32) for a in (w, g, m, v, ve)]
    n = arrs[0].size
    outs = [np.zeros(n, np.float32) for _ in range(4)]
    rc = lib().orc_update_elements_n(ctypes.byref(hp), t, n, *map(_p, arrs), *map(_p, outs))
    if rc != 0:
        raise ValueError("invalid hyper-parameters or step")
    return tuple(outs)


def step_elements(hp: HParams, t: int, wdt: int, gdt: int, mdt: int, w, g, m, v, ve,
                  gidx=None, gidx0: int = 0, e_cur: int = 0, e_next: int = 0) -> float:
    """One step over host arrays updated in place; returns max |updated w|
    (finite values; meaningful for E4M3 storage)."""
    for a in (w, g, m, v, ve):
        assert a.flags.c_contiguous
    n = w.size
    idx = None if gidx is None else _c(gidx, np.int64)
    amax = ctypes.c_float(0.0)
    rc = lib().orc_step_elements(
        n, None if idx is None else _p(idx), gidx0, wdt, gdt, mdt,
        _p(w), _p(g), _p(m), _p(v), _p(ve), ctypes.byref(hp), t, e_cur, e_next,
        ctypes.byref(amax))
    if rc != 0:
        raise ValueError("invalid arguments")
    return float(amax.value)


def fp16_pow2(k: int) -> int:
    """FP16 bits of 2^k, k clamped to [-24, 15]."""
    return int(lib().orc_fp16_pow2(int(k)))


def fp16_decode(h) -> np.ndarray:
    return np.array([lib().orc_fp16_decode(int(x)) for x in np.atleast_1d(h)], np.float32)


def block_exponent(amax: float, k_old: int) -> int:
    return int(lib().orc_block_exponent(ctypes.c_float(amax), int(k_old)))


def step_block_e4m3(hp: HParams, t: int, gdt: int, mdt: int, q, bscale, g, m, v, ve, gidx0: int = 0) -> None:
    """One step of a whole tensor with per-32-block FP16 power-of-two scales;
    q (uint8 codes), bscale (uint16 FP16 bits) and the moments update in place."""
    for a in (q, bscale, g, m, v, ve):
        assert a.flags.c_contiguous
    assert bscale.size == -(-q.size // BLOCK)
    rc = lib().orc_step_block_e4m3(q.size, gidx0, gdt, mdt, _p(q), _p(bscale), _p(g), _p(m), _p(v), _p(ve),
                                   ctypes.byref(hp), t)
    if rc != 0:
        raise ValueError("invalid arguments")


def dequant_bf16(q, e: int = 0, bscale=None) -> np.ndarray:
    """BF16 compute copy of stored E4M3 weights (per-tensor 2^e, or per-block scales)."""
    q = _c(q, np.uint8)
    out = np.zeros(q.size, np.uint16)
    bs = None if bscale is None else _c(bscale, np.uint16)
    lib().orc_dequant_bf16(q.size, _p(q), int(e), None if bs is None else _p(bs), _p(out))
    return out


def e2m1_rne(x) -> np.ndarray:
    return np.array([lib().orc_e2m1_rne(float(v)) for v in np.atleast_1d(np.asarray(x, np.float32))], np.uint8)


def e2m1_sr(x, r32) -> np.ndarray:
    xs = np.atleast_1d(np.asarray(x, np.float32))
    rs = np.atleast_1d(np.asarray(r32, np.uint32))
    return np.array([lib().orc_e2m1_sr(float(v), int(r)) for v, r in zip(xs, rs)], np.uint8)


def e2m1_decode(c) -> np.ndarray:
    return np.array([lib().orc_e2m1_decode(int(v)) for v in np.atleast_1d(c)], np.float32)


def nvfp4_scale_code(amax: float, G: float, c_old: int) -> int:
    return int(lib().orc_nvfp4_scale_code(ctypes.c_float(amax), ctypes.c_float(G), int(c_old)))


def nvfp4_unpack(q, n: int) -> np.ndarray:
    """Codes of n elements from packed bytes (even element in the low nibble)."""
    q = np.asarray(q, np.uint8)
    out = np.empty(2 * q.size, np.uint8)
    out[0::2] = q & 0x0F
    out[1::2] = q >> 4
    return out[:n]


def nvfp4_pack(codes) -> np.ndarray:
    c = np.asarray(codes, np.uint8)
    if c.size % 2:
        c = np.concatenate([c, np.zeros(1, np.uint8)])
    return (c[0::2] & 0x0F) | (c[1::2] << 4)


def step_nvfp4(hp: HParams, t: int, gdt: int, mdt: int, n: int, q, bscale, G: float, g, m, v, ve,
               gidx0: int = 0) -> None:
    """One step of a whole NVFP4 tensor of n elements: q (packed codes),
    bscale (E4M3 block-scale codes) and the moments update in place."""
    for a in (q, bscale, g, m, v, ve):
        assert a.flags.c_contiguous
    assert q.size == (n + 1) // 2 and bscale.size == -(-n // FP4_BLOCK)
    rc = lib().orc_step_nvfp4(n, gidx0, gdt, mdt, _p(q), _p(bscale), ctypes.c_float(G), _p(g), _p(m), _p(v),
                              _p(ve), ctypes.byref(hp), t)
    if rc != 0:
        raise ValueError("invalid arguments")


def dequant_nvfp4_bf16(n: int, q, bscale, G: float) -> np.ndarray:
    q = _c(q, np.uint8)
    bs = _c(bscale, np.uint8)
    out = np.zeros(n, np.uint16)
    lib().orc_dequant_nvfp4_bf16(n, _p(q), _p(bs), ctypes.c_float(G), _p(out))
    return out


class ToyConfig(ctypes.Structure):
    _fields_ = [("mode", ctypes.c_int32), ("split", ctypes.c_int32), ("batch", ctypes.c_int32),
                ("pad", ctypes.c_int32), ("lr_add", ctypes.c_float), ("lr_mul", ctypes.c_float),
                ("rmax", ctypes.c_float), ("tau", ctypes.c_float), ("c_lo", ctypes.c_float),
                ("c_hi", ctypes.c_float), ("seed", ctypes.c_uint64)]


TOY_MODES = {"additive": 0, "multiplicative": 1, "combined": 2}


def toy_config(mode, *, lr_add=0.0, lr_mul=0.0, batch=65536, c_lo=1.0, c_hi=None, split=False, seed=0,
               rmax=0.75, tau=1e-8) -> ToyConfig:
    return ToyConfig(TOY_MODES[mode] if isinstance(mode, str) else mode, int(split), batch, 0, lr_add, lr_mul,
                     rmax, tau, c_lo, c_lo if c_hi is None else c_hi, seed)


def tree_sum(x) -> float:
    x = _c(x, np.float64)
    return float(lib().orc_tree_sum(x.size, _p(x)))


def toy_step(cfg: ToyConfig, w, wstar, t: int) -> float:
    """One toy-diagnostic step: w (uint16 BF16 bits) updated in place; returns
    the minibatch loss before the update."""
    assert w.dtype == np.uint16 and w.flags.c_contiguous
    n, B = w.size, cfg.batch
    if n & (n - 1) or B & (B - 1) or B < 64 or cfg.mode not in (0, 1, 2) or cfg.split not in (0, 1):
        raise ValueError("invalid arguments")
    ws = _c(wstar, np.float32)
    return float(lib().orc_toy_step(ctypes.byref(cfg), n, _p(w), _p(ws), t))


def global_offsets(numels) -> List[int]:
    """First global element index of each tensor: the previous tensor's end
    rounded up to a multiple of 8."""
    offs, o = [], 0
    for n in numels:
        offs.append(o)
        o = -(-(o + int(n)) // ALIGN) * ALIGN
    return offs


def fp8_init(tensors, exps: Sequence[int]) -> List[list]:
    """Per-tensor FP8 state [exponent, amax] before the first step: amax is the
    largest |decoded stored weight|."""
    return [[int(e), e4m3_amax(t["w"], int(e))] for t, e in zip(tensors, exps)]


def step(tensors, *, wdt, gdt: int, mdt: int, hp: HParams, t: int,
         fp8_state: Optional[List[list]] = None) -> None:
    """One optimizer step over a tensor list.  tensors: list of dicts of 1-D
    numpy arrays w, g, m, v, ve (updated in place).  wdt is the weight format
    of every tensor, or a list with one format per tensor.  For E4M3 storage,
    fp8_state[k] = [exponent the stored weights use, largest |w| before this
    step]; it is advanced in place: the weights are re-encoded with the
    exponent chosen from that largest |w|, and the new largest |w| is recorded.
    For E4M3_B32 storage the dict also holds "bscale" (FP16 block scales,
    updated in place); for NVFP4 storage "w" holds packed codes, "bscale" the
    E4M3 block-scale codes (updated in place) and "gscale" the tensor scale."""
    offs = global_offsets([d["g"].size for d in tensors])   # element counts (NVFP4 "w" is packed)
    formats = list(wdt) if isinstance(wdt, (list, tuple)) else [wdt] * len(tensors)
    for k, d in enumerate(tensors):
        wdt = formats[k]
        if d["g"].size == 0:
            continue
        if wdt == E4M3_B32:
            step_block_e4m3(hp, t, gdt, mdt, d["w"], d["bscale"], d["g"], d["m"], d["v"], d["ve"],
                            gidx0=offs[k])
        elif wdt == NVFP4:
            step_nvfp4(hp, t, gdt, mdt, d["g"].size, d["w"], d["bscale"], d["gscale"], d["g"], d["m"],
                       d["v"], d["ve"], gidx0=offs[k])
        elif wdt == E4M3:
            e_cur, a_cur = fp8_state[k]
            e_next = fp8_next_exponent(a_cur, e_cur)
            a_next = step_elements(hp, t, wdt, gdt, mdt, d["w"], d["g"], d["m"], d["v"], d["ve"],
                                   gidx0=offs[k], e_cur=e_cur, e_next=e_next)
            fp8_state[k][0] = e_next
            fp8_state[k][1] = a_next
        else:
            step_elements(hp, t, wdt, gdt, mdt, d["w"], d["g"], d["m"], d["v"], d["ve"],
                          gidx0=offs[k])
