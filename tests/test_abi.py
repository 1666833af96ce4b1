"""The C-ABI library: it builds for sm_103a, loads, exports every entry point
include/mpadam.h declares, and rejects bad arguments on the host (these
checks run before any CUDA call, so they need no GPU)."""
import ctypes
import math
import re
from pathlib import Path

import pytest

from paper_2607_10611_gb300 import builder as B

ROOT = Path(__file__).resolve().parents[1]


@pytest.fixture(scope="module")
def N():
    B.build()
    from paper_2607_10611_gb300 import _native
    return _native


def declared_functions():
    text = (ROOT / "include" / "mpadam.h").read_text()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(mpadam_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for must in ("mpadam_create", "mpadam_step", "mpadam_destroy", "mpadam_last_error"):
        assert must in names


def test_library_exports_every_declared_symbol(N):
    lib = ctypes.CDLL(str(B.LIB))
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert sorted(N.EXPORTED) == declared_functions()


def test_library_is_built_for_sm_103a_only():
    assert "arch=compute_103a,code=sm_103a" in " ".join(B.NVCC_FLAGS)
    assert B.LIB.exists()


def _tensor_tuple(n=16):
    return [(0x1000, 0x2000, 0x3000, 0x4000, n)]


@pytest.mark.parametrize("field,value", [
    ("eps", 0.0), ("eps", -1.0), ("tau", 0.0), ("beta1", 1.0), ("beta2", -0.1),
    ("lr_add", -1e-3), ("lr_mul", math.nan), ("rmax_neg", 1.0), ("rmax_pos", 0.0),
    ("g_max", 0.0), ("dmult_max", -1.0), ("w_max", 0.0), ("wd_add", -0.1),
    ("weight_dtype", 0), ("grad_dtype", 2), ("moment_dtype", 2), ("rounding", 2),
    ("bias_correction", 3), ("reserved", 1)])
def test_create_rejects_bad_config(N, field, value):
    cfg = N.make_config(**{field: value})
    with pytest.raises(N.MPAdamError) as ei:
        N.mpadam_create(_tensor_tuple(), cfg)
    assert ei.value.status == N.MPADAM_EINVAL
    assert N.mpadam_last_error()


def test_create_rejects_bad_tensors(N):
    cfg = N.make_config()
    for bad in ([(0, 0x2000, 0x3000, 0x4000, 8)],            # NULL w
                [(0x1001, 0x2000, 0x3000, 0x4000, 8)],       # misaligned bf16 w
                [(0x1000, 0x2002, 0x3000, 0x4000, 8)],       # misaligned fp32 moment
                [(0x1000, 0x2000, 0x3000, 0x4000, -1)]):     # negative size
        with pytest.raises(N.MPAdamError) as ei:
            N.mpadam_create(bad, cfg)
        assert ei.value.status == N.MPADAM_EINVAL


def test_e4m3_requires_scale_rings(N):
    cfg = N.make_config(weight_dtype="e4m3")
    with pytest.raises(N.MPAdamError) as ei:
        N.mpadam_create(_tensor_tuple(), cfg)
    assert "fp8" in str(ei.value)


def test_null_state_and_bad_step(N):
    lib = N.lib()
    assert lib.mpadam_step(None, None, 1, None) == N.MPADAM_EINVAL
    assert lib.mpadam_destroy(None) == N.MPADAM_OK
    assert lib.mpadam_rng_lanes(0, 1, 7, 0, 4, None, None) == N.MPADAM_EINVAL
    assert lib.mpadam_rng_lanes(0, 1, N.MPADAM_BF16, -1, 4, None, None) == N.MPADAM_EINVAL
    assert lib.mpadam_set_tail_pool(None, 768, 4) == N.MPADAM_EINVAL
    assert lib.mpadam_set_grid(None, 0) == N.MPADAM_EINVAL


def test_create_ex_rejects_bad_lists_on_the_host(N):
    """Per-tensor formats, block scales, compute copies and tensor scales are
    validated before any CUDA call."""
    cfg = N.make_config()
    W, M, S, C = 0x10000, 0x20000, 0x30000, 0x40000
    bad = [
        (W, M, M, M, 64, 9, 0, 0),                    # unknown format
        (W, M, M, M, 64, "e4m3_b32", 0, 0),           # block scales missing
        (W, M, M, M, 64, "e4m3_b32", S + 1, 0),       # misaligned FP16 scales
        (W, M, M, M, 64, "nvfp4", 0, 0, 1e-3),        # NVFP4 scales missing
        (W, M, M, M, 64, "nvfp4", S, 0, 0.0),         # no tensor scale
        (W, M, M, M, 64, "nvfp4", S, 0, float("nan")),
        (W, M, M, M, 64, "bf16", 0, C),               # compute copy of BF16 weights
        (W, M, M, M, 64, "bf16", S, 0),               # block scales on BF16 weights
        (W, M, M, M, 64, "e4m3_b32", S, 0, 1e-3),     # tensor scale on another format
        (W, M, M, M, 64, "e4m3", 0, 0),               # E4M3 without the fp8 rings
        (W, M, M + 2, M, 64, "bf16", 0, 0),           # misaligned fp32 moment
    ]
    for t in bad:
        with pytest.raises(N.MPAdamError) as ei:
            N.mpadam_create_ex([t], cfg)
        assert ei.value.status == N.MPADAM_EINVAL, t
    for fmt in ("e4m3_b32", "nvfp4"):  # the uniform entry point cannot carry block scales
        with pytest.raises(N.MPAdamError):
            N.mpadam_create(_tensor_tuple(), N.make_config(weight_dtype=fmt))


def test_toy_create_rejects_bad_config_on_the_host(N):
    ok = dict(mode=2, split=0, batch=64, reserved=0, lr_add=1.0, lr_mul=1.0, rmax=0.75, tau=1e-8, c_lo=1.0,
              c_hi=1.0, seed=0)
    for n, over in [(100, {}), (32, {}), (1 << 31, {}), (64, {"batch": 48}), (64, {"batch": 32, "split": 1}),
                    (64, {"batch": 1 << 17}), (64, {"mode": 3}), (64, {"split": 2}), (64, {"tau": 0.0}),
                    (64, {"lr_add": -1.0}), (64, {"lr_mul": float("inf")}), (64, {"reserved": 1}),
                    (64, {"c_lo": float("nan")})]:
        with pytest.raises(N.MPAdamError) as ei:
            N.mpadam_toy_create(n, N.mpadam_toy_config(**{**ok, **over}))
        assert ei.value.status == N.MPADAM_EINVAL, (n, over)
    lib = N.lib()
    assert lib.mpadam_toy_step(None, None, None, 1, None, None) == N.MPADAM_EINVAL
    assert lib.mpadam_toy_run(None, None, None, 1, 1, None, None) == N.MPADAM_EINVAL
    assert lib.mpadam_toy_destroy(None) == N.MPADAM_OK
    assert lib.mpadam_host_buffer_alloc(0, None) == N.MPADAM_EINVAL
    assert lib.mpadam_host_buffer_free(None, 16) == N.MPADAM_OK
