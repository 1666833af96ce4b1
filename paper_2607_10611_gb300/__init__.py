"""GB300-native fused M+Adam optimizer step (arxiv 2607.10611).

The step runs in one hand-written sm_103a CUDA kernel behind the C ABI of
include/mpadam.h; this package holds that library's sources (csrc/), its
build script and a thin ctypes binding with the C entry points' names.
PyTorch is used only for device memory and streams.
"""
from .builder import build  # noqa: F401

__all__ = ["build", "native", "MPAdam"]


def __getattr__(name):
    if name == "native":
        from . import _native
        return _native
    if name == "MPAdam":
        from .optimizer import MPAdam
        return MPAdam
    raise AttributeError(name)
