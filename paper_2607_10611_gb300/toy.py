"""The BF16-stored matrix-fitting diagnostic (the toy diagnostic of Sec. 5.1
and its appendix) on torch tensors: argument marshalling around
mpadam_toy_create / mpadam_toy_step (no arithmetic here).
"""
from __future__ import annotations

import math
from typing import Optional

import torch

from . import _native as N


class ToyDiagnostic:
    """Minimise c ||W - W*||^4 over BF16-stored W with one of the three
    update rules (``mode``: "additive", "multiplicative", "combined").
    ``w`` (bfloat16) and ``wstar`` (float32) are flat CUDA tensors of a
    power-of-two length; ``w`` is updated in place by every step."""

    def __init__(self, w: torch.Tensor, wstar: torch.Tensor, *, mode: str, lr_add: float = 0.0,
                 lr_mul: float = 0.0, batch: int = 65536, c_lo: float = 1.0, c_hi: Optional[float] = None,
                 split: bool = False, seed: int = 0, rmax: float = 0.75, tau: float = 1e-8):
        for t, dt in ((w, torch.bfloat16), (wstar, torch.float32)):
            if t.dtype != dt or not t.is_cuda or not t.is_contiguous():
                raise ValueError(f"expected a contiguous CUDA tensor of {dt}")
        if w.numel() != wstar.numel():
            raise ValueError("w and wstar differ in size")
        self.w, self.wstar = w, wstar
        cfg = N.mpadam_toy_config(N.TOY_MODES[mode], int(split), batch, 0, lr_add, lr_mul, rmax, tau, c_lo,
                                  c_lo if c_hi is None else c_hi, seed)
        with torch.cuda.device(w.device):
            self.state = N.mpadam_toy_create(w.numel(), cfg)
        self.loss = torch.zeros(1, dtype=torch.float64, device=w.device)

    def step(self, t: int, loss_out: Optional[torch.Tensor] = None, stream: Optional[torch.cuda.Stream] = None):
        """Step t; the minibatch loss (before the update) goes to loss_out
        (a CUDA float64 element) or to self.loss."""
        s = (stream or torch.cuda.current_stream(self.w.device)).cuda_stream
        out = self.loss if loss_out is None else loss_out
        N.mpadam_toy_step(self.state, self.w.data_ptr(), self.wstar.data_ptr(), t, out.data_ptr(), s)

    def run(self, first_step: int, steps: int, losses: Optional[torch.Tensor] = None,
            stream: Optional[torch.cuda.Stream] = None):
        """Steps first_step .. first_step + steps - 1 (CUDA-graph replays);
        losses: a CUDA float64 tensor of `steps` elements, or None."""
        s = (stream or torch.cuda.current_stream(self.w.device)).cuda_stream
        N.mpadam_toy_run(self.state, self.w.data_ptr(), self.wstar.data_ptr(), first_step, steps,
                         losses.data_ptr() if losses is not None else 0, s)

    def close(self):
        if getattr(self, "state", None):
            N.mpadam_toy_destroy(self.state)
            self.state = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
