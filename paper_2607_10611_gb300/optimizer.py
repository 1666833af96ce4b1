"""MPAdam: torch-tensor marshalling around the C ABI (no arithmetic here).

Holds references to the caller's device tensors (weights, moments) so their
memory outlives the native state, allocates the E4M3 scale rings with torch,
and forwards every step to mpadam_step on the current torch stream.
"""
from __future__ import annotations

from typing import List, Optional, Sequence

import torch

from . import _native as N

_STORAGE = {"bf16": torch.bfloat16, "e4m3": torch.uint8, "f32": torch.float32}


class MPAdam:
    def __init__(self, w: Sequence[torch.Tensor], m: Sequence[torch.Tensor], v: Sequence[torch.Tensor],
                 ve: Sequence[torch.Tensor], *, weight_dtype: str = "bf16", grad_dtype: str = "f32",
                 moment_dtype: str = "f32", rounding: str = "nearest", seed: int = 0,
                 fp8_exp: Optional[Sequence[int]] = None, first_step: int = 1, **hparams):
        self.w, self.m, self.v, self.ve = list(w), list(m), list(v), list(ve)
        self.weight_dtype, self.grad_dtype, self.moment_dtype = weight_dtype, grad_dtype, moment_dtype
        for t, dt in [(x, weight_dtype) for x in self.w] + \
                     [(x, moment_dtype) for x in self.m + self.v + self.ve]:
            if t.dtype != _STORAGE[dt] or not t.is_cuda or not t.is_contiguous():
                raise ValueError(f"expected contiguous CUDA tensors of {_STORAGE[dt]}")
        self.n = len(self.w)
        self.cfg = N.make_config(weight_dtype=weight_dtype, grad_dtype=grad_dtype,
                                 moment_dtype=moment_dtype, rounding=rounding, seed=seed, **hparams)
        dev = self.w[0].device if self.n else torch.device("cuda", torch.cuda.current_device())
        self.fp8_exp_ring = self.fp8_amax_ring = None
        if weight_dtype == "e4m3":
            self.fp8_exp_ring = torch.zeros(2 * max(1, self.n), dtype=torch.int32, device=dev)
            self.fp8_amax_ring = torch.zeros(3 * max(1, self.n), dtype=torch.int32, device=dev)
        with torch.cuda.device(dev):
            self.state = N.mpadam_create(
                [(a.data_ptr(), b.data_ptr(), c.data_ptr(), d.data_ptr(), a.numel())
                 for a, b, c, d in zip(self.w, self.m, self.v, self.ve)], self.cfg,
                self.fp8_exp_ring.data_ptr() if self.fp8_exp_ring is not None else 0,
                self.fp8_amax_ring.data_ptr() if self.fp8_amax_ring is not None else 0)
            if weight_dtype == "e4m3":
                if fp8_exp is None:
                    raise ValueError("E4M3 weights need the exponents they are stored with (fp8_exp)")
                N.mpadam_fp8_init(self.state, list(fp8_exp), first_step,
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
