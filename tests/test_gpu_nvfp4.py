"""GPU parity of NVFP4 master weights (E2M1 codes, an E4M3 scale per 16
elements, a binary32 tensor scale; current block scaling) and of their BF16
compute copy: every stored bit against the oracle (packed codes, block-scale
codes, moments, compute copies), alone and in lists that mix all four weight
formats (Sec. 5.2's NVFP4 master weights)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W

pytestmark = pytest.mark.gpu

EDGE_SIZES = (0, 1, 7, 8, 9, 15, 16, 17, 31, 33, 2047, 3840, 3841, 4097, 0, 3, 65536 + 5)


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2607_10611_gb300 import build
    build()


def P():
    import parity
    return parity


def _fp4(gd="f32", md="f32", rnd="stochastic", cc=True, sizes=EDGE_SIZES, formats=()):
    specs = tuple(W.TensorSpec(f"t{i}", n, "matrix") for i, n in enumerate(sizes))
    return W.Workload(name="fp4", specs=specs, weight_dtype="nvfp4", grad_dtype=gd, moment_dtype=md,
                      rounding=rnd, steps=3, seed=17, zero_frac=0.05, grad=("normal_logu", 1e-6, 1e-1),
                      compute_copy=cc, format_list=tuple(formats))


def _run_steps(r, steps, what):
    p = P()
    for t in range(1, steps + 1):
        r.step(t)
        res = r.compare(t + 1)
        assert res["contract_ok"]
        p.assert_exact(res, f"{what} step {t}")


@pytest.mark.parametrize("gd", ["f32", "bf16"])
@pytest.mark.parametrize("md", ["f32", "bf16"])
@pytest.mark.parametrize("rnd", ["nearest", "stochastic"])
def test_nvfp4_every_format_combination(gd, md, rnd):
    r = P().Run(_fp4(gd, md, rnd), warm=True)
    try:
        _run_steps(r, 3, f"nvfp4/{gd}/{md}/{rnd}")
    finally:
        r.close()


def test_nvfp4_without_compute_copy_cold_state():
    r = P().Run(_fp4(cc=False))
    try:
        _run_steps(r, 3, "no compute copy")
    finally:
        r.close()


@pytest.mark.parametrize("misalign", [1, 3])
def test_nvfp4_misaligned_arrays(misalign):
    r = P().Run(_fp4(), warm=True, misalign=misalign)
    try:
        _run_steps(r, 2, f"misalign {misalign}")
    finally:
        r.close()


def test_mixed_list_all_four_formats():
    sizes = (4097, 65, 3840, 1, 0, 20000, 33, 7681, 512, 3, 17, 3841)
    fmts = ("bf16", "nvfp4", "e4m3", "e4m3_b32", "nvfp4", "e4m3", "bf16", "nvfp4", "e4m3_b32", "bf16",
            "nvfp4", "e4m3_b32")
    r = P().Run(_fp4(sizes=sizes, formats=fmts), warm=True)
    try:
        _run_steps(r, 4, "four formats")
    finally:
        r.close()


@pytest.mark.parametrize("layout", ["separate", "flat"])
def test_paper_nvfp4_regime_small(layout):
    r = P().Run(W.SMALL["llama_1p5b_nvfp4"], warm=True, layout=layout)
    try:
        _run_steps(r, 4, f"llama nvfp4 {layout}")
    finally:
        r.close()


@pytest.mark.parametrize("hp", [
    dict(g_max=0.7), dict(w_max=0.03), dict(wd_add=0.1), dict(dmult_max=0.02), dict(bias_correction=0),
    dict(lr_mul=0.0), dict(lr_mul=0.5, lr_add=0.05), dict(eps=1e-10), dict(lr_mul=5.0),
])
def test_nvfp4_algorithm2_options(hp):
    r = P().Run(W.SMALL["llama_1p5b_nvfp4"], warm=True, hp=hp)
    try:
        _run_steps(r, 3, f"{hp}")
    finally:
        r.close()


@pytest.mark.parametrize("lr", [1e-7, 1e-5, 3e-2])
def test_nvfp4_block_maxima_at_the_top_code(lr):
    """Every block holds an element at +-6 (the top E2M1 code), so small
    updates put the block maximum at the edge of its scale's range: scales
    that stay, scales that step up, and undecided bounds."""
    p = P()
    wl = W.replace(_fp4(sizes=(3840 * 3, 4097, 97)), rounding="nearest", zero_frac=0.0)
    mt = W.materialize(wl, "cpu", warm_state=True)
    rng = np.random.default_rng(1)
    for k in range(len(mt.w)):
        n = mt.g[k].numel()
        codes = oracle.nvfp4_unpack(W.to_numpy_bits(mt.w[k]), n)
        top = np.arange(0, n, 16) + rng.integers(0, 16, (n + 15) // 16)
        top = top[top < n]
        codes[top] = np.where(rng.random(top.size) < 0.5, 7, 15)
        mt.w[k].copy_(torch.from_numpy(oracle.nvfp4_pack(codes)))
    r = p.Run(wl, mt=mt, hp=dict(lr_add=lr, lr_mul=lr))
    try:
        before = [b.clone() for b in r.dev["bscale"]]
        _run_steps(r, 3, f"top codes lr={lr}")
        changed = sum(int((a != b).sum()) for a, b in zip(before, r.dev["bscale"]))
        assert changed > 0
    finally:
        r.close()


@pytest.mark.parametrize("md", ["bf16", "f32"])
def test_nvfp4_nan_inf_and_odd_scales(md):
    """Non-finite inputs and odd block scales send elements to the exact
    branch: re-read from the stage (BF16 moments) or from global memory
    (binary32 moments, the stage already released)."""
    p = P()
    wl = _fp4(md=md)
    mt = W.materialize(wl, "cpu", warm_state=True)
    big = max(range(len(mt.g)), key=lambda k: mt.g[k].numel())
    g = mt.g[big]
    g[::97] = float("nan")
    g[5::131] = float("inf")
    g[7::151] = -float("inf")
    mt.ve[big][17::191] = float("inf")
    bs = mt.bscale[big]
    bs[3] = 0x00   # zero scale
    bs[4] = 0x7F   # NaN scale
    bs[5] = 0x80   # negative zero
    bs[6] = 0xFE   # -448
    bs[7] = 0x01   # smallest subnormal E4M3
    bs[8] = 0x7E   # 448
    r = p.Run(wl, mt=mt)
    try:
        _run_steps(r, 2, "non-finite")
    finally:
        r.close()


def test_nvfp4_tiny_and_huge_tensor_scales():
    """Tensor scales whose block step d = s * G leaves the range the fast
    division covers: the exact division runs, same bits."""
    p = P()
    wl = _fp4(sizes=(4097, 100))
    mt = W.materialize(wl, "cpu", warm_state=True)
    mt.gscale[0] = 2.0 ** -130
    mt.gscale[1] = 2.0 ** 100
    r = p.Run(wl, mt=mt)
    try:
        _run_steps(r, 2, "tensor scales")
    finally:
        r.close()


def test_nvfp4_grid_size_does_not_change_results():
    p = P()
    runs = []
    for grid in (0, 1, 7, 333):
        r = p.Run(W.SMALL["llama_1p5b_nvfp4"], warm=True)
        if grid:
            r.opt.set_grid(grid)
        for t in range(1, 3):
            r.step(t)
        runs.append(r)
    for r in runs:
        p.assert_exact(r.compare(3), "grid")
    for r in runs:
        r.close()


def test_create_ex_rejects_bad_nvfp4():
    from paper_2607_10611_gb300 import _native as N
    w8 = torch.zeros(32, dtype=torch.uint8, device="cuda")
    m = torch.zeros(64, device="cuda")
    sc = torch.ones(4, dtype=torch.uint8, device="cuda")
    cfg = N.make_config()
    P_ = lambda t: t.data_ptr()
    bad = [
        [(P_(w8), P_(m), P_(m), P_(m), 64, "nvfp4", 0, 0, 1e-3)],          # block scales missing
        [(P_(w8), P_(m), P_(m), P_(m), 64, "nvfp4", P_(sc), 0, 0.0)],       # no tensor scale
        [(P_(w8), P_(m), P_(m), P_(m), 64, "nvfp4", P_(sc), 0, -1.0)],      # negative tensor scale
        [(P_(w8), P_(m), P_(m), P_(m), 64, "nvfp4", P_(sc), 0, float("inf"))],
        [(P_(w8), P_(m), P_(m), P_(m), 64, "e4m3_b32", P_(sc), 0, 1e-3)],   # tensor scale on another format
    ]
    for tensors in bad:
        with pytest.raises(N.MPAdamError):
            N.mpadam_create_ex(tensors, cfg)
    with pytest.raises(N.MPAdamError):   # NVFP4 needs mpadam_create_ex
        N.mpadam_create([(P_(w8), P_(m), P_(m), P_(m), 64)], N.make_config(weight_dtype="nvfp4"))
