"""MPAdam: torch-tensor marshalling around the C ABI (no arithmetic here).

Holds references to the caller's device tensors (weights, moments, block
scales, compute copies) so their memory outlives the native state, allocates
the E4M3 scale rings with torch, and forwards every step to mpadam_step on
the current torch stream.  `weight_dtype` is one format for the whole list
("bf16", "e4m3") or a list with one format per tensor ("bf16", "e4m3",
"e4m3_b32", "nvfp4"); the latter, block scales or compute copies go through
mpadam_create_ex.  NVFP4 weights are packed bytes (two codes each), so the
element count of every tensor is taken from its first moment.
"""
from __future__ import annotations

from typing import List, Optional, Sequence

import torch

from . import _native as N

_STORAGE = {"bf16": torch.bfloat16, "e4m3": torch.uint8, "e4m3_b32": torch.uint8, "nvfp4": torch.uint8,
            "f32": torch.float32}
_SCALES = {"e4m3_b32": torch.float16, "nvfp4": torch.uint8}


class HostBuffer:
    """Page-locked, huge-page host memory from mpadam_host_buffer_alloc, as a
    1-D CPU tensor of `dtype` (for mpadam_step_host's gradients and weights)."""

    def __init__(self, numel: int, dtype: torch.dtype):
        import ctypes
        import numpy as np
        itemsize = torch.empty(0, dtype=dtype).element_size()
        self.nbytes = max(1, numel * itemsize)
        self.ptr = N.mpadam_host_buffer_alloc(self.nbytes)
        raw = (ctypes.c_uint8 * self.nbytes).from_address(self.ptr)
        self.tensor = torch.from_numpy(np.frombuffer(raw, dtype=np.uint8)).view(dtype)[:numel]

    def free(self):
        if getattr(self, "ptr", None):
            self.tensor = None
            N.mpadam_host_buffer_free(self.ptr, self.nbytes)
            self.ptr = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


class MPAdam:
    def __init__(self, w: Sequence[torch.Tensor], m: Sequence[torch.Tensor], v: Sequence[torch.Tensor],
                 ve: Sequence[torch.Tensor], *, weight_dtype="bf16", grad_dtype: str = "f32",
                 moment_dtype: str = "f32", rounding: str = "nearest", seed: int = 0,
                 fp8_exp: Optional[Sequence[int]] = None, first_step: int = 1,
                 block_scales: Optional[Sequence[Optional[torch.Tensor]]] = None,
                 compute: Optional[Sequence[Optional[torch.Tensor]]] = None,
                 global_scales: Optional[Sequence[float]] = None, **hparams):
        self.w, self.m, self.v, self.ve = list(w), list(m), list(v), list(ve)
        self.n = len(self.w)
        per_tensor = not isinstance(weight_dtype, str)
        self.formats = list(weight_dtype) if per_tensor else [weight_dtype] * self.n
        self.block_scales = list(block_scales) if block_scales is not None else [None] * self.n
        self.compute = list(compute) if compute is not None else [None] * self.n
        self.global_scales = [float(x or 0.0) for x in global_scales] if global_scales is not None else [0.0] * self.n
        if not (len(self.formats) == len(self.block_scales) == len(self.compute) == len(self.global_scales) == self.n):
            raise ValueError("one weight format, block-scale and compute entry per tensor")
        self.weight_dtype, self.grad_dtype, self.moment_dtype = weight_dtype, grad_dtype, moment_dtype
        for t, dt in [(x, f) for x, f in zip(self.w, self.formats)] + \
                     [(x, moment_dtype) for x in self.m + self.v + self.ve] + \
                     [(x, "bf16") for x in self.compute if x is not None]:
            if t.dtype != _STORAGE[dt] or not t.is_cuda or not t.is_contiguous():
                raise ValueError(f"expected contiguous CUDA tensors of {_STORAGE[dt]}")
        for x, f in zip(self.block_scales, self.formats):
            if x is not None and (x.dtype != _SCALES.get(f) or not x.is_cuda or not x.is_contiguous()):
                raise ValueError("block scales must be contiguous CUDA tensors (float16 for e4m3_b32, "
                                 "uint8 E4M3 codes for nvfp4)")
        extended = per_tensor or any(x is not None for x in self.block_scales + self.compute)
        uniform = weight_dtype if not per_tensor else "bf16"
        self.cfg = N.make_config(weight_dtype="bf16" if extended else uniform, grad_dtype=grad_dtype,
                                 moment_dtype=moment_dtype, rounding=rounding, seed=seed, **hparams)
        dev = self.w[0].device if self.n else torch.device("cuda", torch.cuda.current_device())
        self.fp8_exp_ring = self.fp8_amax_ring = None
        any_e4m3 = "e4m3" in self.formats or (not self.n and weight_dtype == "e4m3")
        if any_e4m3:
            self.fp8_exp_ring = torch.zeros(2 * max(1, self.n), dtype=torch.int32, device=dev)
            self.fp8_amax_ring = torch.zeros(3 * max(1, self.n), dtype=torch.int32, device=dev)
        rings = (self.fp8_exp_ring.data_ptr() if any_e4m3 else 0, self.fp8_amax_ring.data_ptr() if any_e4m3 else 0)
        ptr = lambda t: t.data_ptr() if t is not None else 0
        with torch.cuda.device(dev):
            if extended:
                self.state = N.mpadam_create_ex(
                    [(a.data_ptr(), b.data_ptr(), c.data_ptr(), d.data_ptr(), b.numel(), f, ptr(bs), ptr(cc), gs)
                     for a, b, c, d, f, bs, cc, gs in zip(self.w, self.m, self.v, self.ve, self.formats,
                                                          self.block_scales, self.compute, self.global_scales)],
                    self.cfg, *rings)
            else:
                self.state = N.mpadam_create(
                    [(a.data_ptr(), b.data_ptr(), c.data_ptr(), d.data_ptr(), a.numel())
                     for a, b, c, d in zip(self.w, self.m, self.v, self.ve)], self.cfg, *rings)
            if "e4m3" in self.formats:
                if fp8_exp is None:
                    raise ValueError("E4M3 weights need the exponents they are stored with (fp8_exp)")
                N.mpadam_fp8_init(self.state, [int(e) for e in fp8_exp], first_step,
                                  torch.cuda.current_stream().cuda_stream)
        self.device = dev

    # -- steps ---------------------------------------------------------------
    def step(self, grads: Sequence[torch.Tensor], t: int, stream: Optional[torch.cuda.Stream] = None):
        s = (stream or torch.cuda.current_stream(self.device)).cuda_stream
        N.mpadam_step(self.state, [g.data_ptr() for g in grads], t, s)

    def step_ptrs(self, grad_ptrs: Sequence[int], t: int, stream: int):
        N.mpadam_step(self.state, grad_ptrs, t, stream)

    def step_host(self, host_grads: Sequence[torch.Tensor], host_w_out: Sequence[torch.Tensor], t: int,
                  stream: Optional[torch.cuda.Stream] = None):
        s = (stream or torch.cuda.current_stream(self.device)).cuda_stream
        N.mpadam_step_host(self.state, [g.data_ptr() for g in host_grads],
                           [w.data_ptr() for w in host_w_out], t, s)

    # -- introspection -------------------------------------------------------
    def fp8_exponents(self, t: int) -> List[int]:
        """Exponents the stored weights use before step t."""
        n = self.n
        return self.fp8_exp_ring[(t % 2) * n:(t % 2) * n + n].tolist()

    def fp8_amax(self, t: int) -> torch.Tensor:
        """Largest |w| recorded for use by step t (binary32)."""
        n = self.n
        return self.fp8_amax_ring[(t % 3) * n:(t % 3) * n + n].view(torch.float32).clone()

    def global_offsets(self) -> List[int]:
        return [N.mpadam_global_offset(self.state, k) for k in range(self.n)]

    def device_status(self) -> int:
        """Device error bits of the steps so far (0 = none); synchronises."""
        return N.mpadam_device_status(self.state)

    def set_grid(self, ctas: int):
        N.mpadam_set_grid(self.state, ctas)

    def set_tail_pool(self, static_q: int, chunk_tiles: int):
        """Static share (in 1/1024) of each CTA's tile run and the pool's chunk length."""
        N.mpadam_set_tail_pool(self.state, static_q, chunk_tiles)

    def launch_info(self):
        return N.mpadam_launch_info(self.state)

    def close(self):
        if getattr(self, "state", None):
            N.mpadam_destroy(self.state)
            self.state = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
