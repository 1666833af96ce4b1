"""GPU parity of block-scaled E4M3 weights (one FP16 power-of-two scale per 32
elements, current scaling), of mixed-format tensor lists (BF16, per-tensor
E4M3 and block-scaled E4M3 in one list, the paper's FP8 regime of Sec. 5.2)
and of the BF16 compute copy written alongside E4M3 master weights: every
stored bit against the oracle (codes, block scales, scale rings, moments,
compute copies)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W

pytestmark = pytest.mark.gpu

EDGE_SIZES = (0, 1, 7, 8, 9, 31, 32, 33, 2047, 3840, 3841, 4097, 0, 3, 65536 + 5)


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2607_10611_gb300 import build
    build()


def P():
    import parity
    return parity


def _blocks(gd="f32", md="f32", rnd="stochastic", cc=True, sizes=EDGE_SIZES, formats=()):
    specs = tuple(W.TensorSpec(f"t{i}", n, "matrix") for i, n in enumerate(sizes))
    return W.Workload(name="blocks", specs=specs, weight_dtype="e4m3_b32", grad_dtype=gd, moment_dtype=md,
                      rounding=rnd, steps=3, seed=13, zero_frac=0.05, grad=("normal_logu", 1e-6, 1e-1),
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
def test_block_scaled_every_format_combination(gd, md, rnd):
    r = P().Run(_blocks(gd, md, rnd), warm=True)
    try:
        _run_steps(r, 3, f"e4m3_b32/{gd}/{md}/{rnd}")
    finally:
        r.close()


def test_block_scaled_without_compute_copy_cold_state():
    r = P().Run(_blocks(cc=False))
    try:
        _run_steps(r, 3, "no compute copy")
    finally:
        r.close()


@pytest.mark.parametrize("misalign", [1, 3])
def test_block_scaled_misaligned_arrays(misalign):
    """Arrays (block scales and compute copies included) shifted off their
    16-byte alignment: element-wise loads and stores, same bits."""
    r = P().Run(_blocks(), warm=True, misalign=misalign)
    try:
        _run_steps(r, 2, f"misalign {misalign}")
    finally:
        r.close()


def test_mixed_list_all_three_formats():
    """BF16, per-tensor E4M3 and block-scaled E4M3 tensors interleaved in one
    list: one launch per format, list-wide global indices and scale rings."""
    sizes = (4097, 65, 3840, 1, 0, 20000, 33, 7681, 512, 3)
    fmts = ("bf16", "e4m3_b32", "e4m3", "e4m3_b32", "e4m3", "e4m3", "bf16", "e4m3_b32", "e4m3", "bf16")
    r = P().Run(_blocks(sizes=sizes, formats=fmts), warm=True)
    try:
        _run_steps(r, 4, "mixed")
    finally:
        r.close()


@pytest.mark.parametrize("layout", ["separate", "flat"])
def test_paper_fp8_regime_small(layout):
    r = P().Run(W.SMALL["llama_1p5b_mixed"], warm=True, layout=layout)
    try:
        _run_steps(r, 4, f"llama mixed {layout}")
    finally:
        r.close()


@pytest.mark.parametrize("hp", [
    dict(g_max=0.7), dict(w_max=0.03), dict(wd_add=0.1), dict(dmult_max=0.02), dict(bias_correction=0),
    dict(lr_mul=0.0), dict(lr_mul=0.5, lr_add=0.05), dict(eps=1e-10), dict(lr_mul=5.0),
])
def test_block_scaled_algorithm2_options(hp):
    r = P().Run(W.SMALL["llama_1p5b_mixed"], warm=True, hp=hp)
    try:
        _run_steps(r, 3, f"{hp}")
    finally:
        r.close()


@pytest.mark.parametrize("lr", [1e-7, 1e-6, 3e-2])
def test_block_maxima_on_scale_thresholds(lr):
    """Every block holds an element at 448 * 2^k of its scale 2^k (the top of
    the E4M3 range), so tiny updates put the block maximum right at the
    threshold where the scale doubles: blocks whose scale is undecided by
    the fast bounds, blocks whose scale changes, and blocks whose scale
    stays.  Large updates change most scales."""
    p = P()
    wl = W.replace(_blocks(sizes=(3840 * 3, 4097, 97)), rounding="nearest", zero_frac=0.0)
    mt = W.materialize(wl, "cpu", warm_state=True)
    rng = np.random.default_rng(1)
    for k in range(len(mt.w)):
        q = mt.w[k]
        n = q.numel()
        top = torch.arange(0, n, 32) + torch.from_numpy(rng.integers(0, 32, (n + 31) // 32))
        top = top[top < n]
        q[top] = torch.where(torch.from_numpy(rng.random(top.numel()) < 0.5), 0x7E, 0xFE).to(torch.uint8)
    r = p.Run(wl, mt=mt, hp=dict(lr_add=lr, lr_mul=lr))
    try:
        before = [b.clone() for b in r.dev["bscale"]]
        _run_steps(r, 3, f"thresholds lr={lr}")
        changed = sum(int((a != b).sum()) for a, b in zip(before, r.dev["bscale"]))
        assert changed > 0
    finally:
        r.close()


def test_block_scaled_nan_inf_and_odd_scales():
    p = P()
    wl = _blocks(md="bf16")
    mt = W.materialize(wl, "cpu", warm_state=True)
    big = max(range(len(mt.g)), key=lambda k: mt.g[k].numel())
    g = mt.g[big]
    g[::97] = float("nan")
    g[5::131] = float("inf")
    g[7::151] = -float("inf")
    mt.w[big][11::173] = 0x7F  # NaN codes
    mt.w[big][12::177] = 0xFF
    mt.ve[big][17::191] = float("inf")
    bs = mt.bscale[big]
    bs[3] = float("inf")                 # a non-finite scale
    bs[4] = 0.0                          # a zero scale
    bs[5] = 3.0                          # not a power of two: decodes as itself, counts as 2^1
    bs[6] = -0.25                        # sign ignored by the exponent, kept by the decode
    bs[7] = 2.0 ** -24                   # smallest subnormal power
    bs[8] = 2.0 ** -15                   # a subnormal power
    r = p.Run(wl, mt=mt)
    try:
        _run_steps(r, 2, "non-finite")
    finally:
        r.close()


def test_block_grid_size_does_not_change_results():
    p = P()
    runs = []
    for grid in (0, 1, 7, 333):
        r = p.Run(W.SMALL["llama_1p5b_mixed"], warm=True)
        if grid:
            r.opt.set_grid(grid)
        for t in range(1, 3):
            r.step(t)
        runs.append(r)
    for r in runs:
        p.assert_exact(r.compare(3), "grid")
    for r in runs:
        r.close()


def test_rng_lanes_of_block_format_are_the_e4m3_lanes():
    from paper_2607_10611_gb300 import _native as N
    n = 4096
    a = torch.zeros(n, dtype=torch.int32, device="cuda")
    b = torch.zeros(n, dtype=torch.int32, device="cuda")
    N.mpadam_rng_lanes(7, 3, N.MPADAM_E4M3_B32, 1000, n, a.data_ptr())
    N.mpadam_rng_lanes(7, 3, N.MPADAM_E4M3, 1000, n, b.data_ptr())
    torch.cuda.synchronize()
    assert torch.equal(a, b)
    want = oracle.rng_lanes(7, 3, np.arange(1000, 1000 + n, dtype=np.uint64), oracle.E4M3)
    np.testing.assert_array_equal(a.cpu().numpy().view(np.uint32), want)


def test_create_ex_rejects_bad_lists():
    from paper_2607_10611_gb300 import _native as N
    w8 = torch.zeros(64, dtype=torch.uint8, device="cuda")
    wb = torch.zeros(64, dtype=torch.bfloat16, device="cuda")
    m = torch.zeros(64, device="cuda")
    sc = torch.ones(2, dtype=torch.float16, device="cuda")
    cc = torch.zeros(64, dtype=torch.bfloat16, device="cuda")
    cfg = N.make_config()
    P_ = lambda t: t.data_ptr()
    bad = [
        [(P_(w8), P_(m), P_(m), P_(m), 64, "e4m3_b32", 0, 0)],            # block scales missing
        [(P_(wb), P_(m), P_(m), P_(m), 64, "bf16", 0, P_(cc))],           # compute copy of BF16 weights
        [(P_(wb), P_(m), P_(m), P_(m), 64, "bf16", P_(sc), 0)],           # scales on BF16 weights
        [(P_(w8), P_(m), P_(m), P_(m), 64, "e4m3", 0, 0)],                # E4M3 without rings
        [(P_(w8), P_(m), P_(m), P_(m), 64, 7, 0, 0)],                     # unknown format
        [(P_(w8), P_(m), P_(m), P_(m), 64, "e4m3_b32", P_(sc) + 1, 0)],   # misaligned scales
    ]
    for tensors in bad:
        with pytest.raises(N.MPAdamError):
            N.mpadam_create_ex(tensors, cfg)
    with pytest.raises(N.MPAdamError):   # block scales need mpadam_create_ex
        N.mpadam_create([(P_(w8), P_(m), P_(m), P_(m), 64)], N.make_config(weight_dtype="e4m3_b32"))
