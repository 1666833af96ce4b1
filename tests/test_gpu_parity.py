"""GPU parity: the CUDA step (through the C ABI) against the oracle, element by
element, on seeded inputs at sizes the oracle finishes in seconds.  Every
stored bit must agree (see tests/parity.py for the tolerance argument)."""
import math

import numpy as np
import pytest
import torch

import oracle
import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2607_10611_gb300 import build
    build()


def P():
    import parity
    return parity


# -----------------------------------------------------------------------------
# The five workloads at small size, several steps, cold and warm states
# -----------------------------------------------------------------------------
@pytest.mark.parametrize("name", list(W.SMALL))
@pytest.mark.parametrize("warm", [False, True])
def test_small_workloads_bit_exact(name, warm):
    p = P()
    r = p.Run(W.SMALL[name], warm=warm)
    try:
        p.assert_exact(r.compare(1), f"{name} before step 1")
        for t in range(1, 5):
            r.step(t)
            res = r.compare(t + 1)
            assert res["contract_ok"]
            p.assert_exact(res, f"{name} step {t}")
    finally:
        r.close()


# Past the first steps: from the zero state of Algorithm 1, the bias
# corrections change with t, the moments grow, and the E4M3 scale rings rotate
# with period 6 (exponent slot t mod 2, amax slot t mod 3).  Twelve steps cover
# two full periods; the GPT-2 list runs its configuration's 100 steps.  Every
# array and both rings are compared after every step.
@pytest.mark.parametrize("name", list(W.SMALL))
def test_small_workloads_many_steps(name):
    p = P()
    steps = 100 if name == "gpt2_124m" else 12
    r = p.Run(W.SMALL[name])
    try:
        for t in range(1, steps + 1):
            r.step(t)
            res = r.compare(t + 1)
            assert res["contract_ok"]
            p.assert_exact(res, f"{name} step {t}")
    finally:
        r.close()


# -----------------------------------------------------------------------------
# Every kernel instance on ragged sizes (tails, tiny tensors, empty tensors)
# -----------------------------------------------------------------------------
EDGE_SIZES = (0, 1, 7, 8, 9, 15, 16, 17, 2047, 2048, 2049, 4097, 0, 3, 65536 + 5)


def _edge_workload(wd, gd, md, rnd):
    specs = tuple(W.TensorSpec(f"t{i}", n, "flat") for i, n in enumerate(EDGE_SIZES))
    return W.Workload(name="edge", specs=specs, weight_dtype=wd, grad_dtype=gd, moment_dtype=md,
                      rounding=rnd, steps=3, seed=11, zero_frac=0.1, grad=("normal_logu", 1e-6, 1e-1))


@pytest.mark.parametrize("wd", ["bf16", "e4m3"])
@pytest.mark.parametrize("gd", ["f32", "bf16"])
@pytest.mark.parametrize("md", ["f32", "bf16"])
@pytest.mark.parametrize("rnd", ["nearest", "stochastic"])
def test_all_format_combinations_on_edge_sizes(wd, gd, md, rnd):
    p = P()
    r = p.Run(_edge_workload(wd, gd, md, rnd), warm=True)
    try:
        for t in range(1, 4):
            r.step(t)
            p.assert_exact(r.compare(t + 1), f"{wd}/{gd}/{md}/{rnd} step {t}")
    finally:
        r.close()


@pytest.mark.parametrize("misalign", [1, 3])
@pytest.mark.parametrize("wd", ["bf16", "e4m3"])
def test_misaligned_tensors_take_the_element_path(misalign, wd):
    p = P()
    r = p.Run(_edge_workload(wd, "f32", "f32", "stochastic"), warm=True, misalign=misalign)
    try:
        for t in range(1, 3):
            r.step(t)
            p.assert_exact(r.compare(t + 1), f"misalign {misalign}")
    finally:
        r.close()


def test_flat_layout_matches():
    p = P()
    r = p.Run(W.SMALL["ragged_20k"], layout="flat", warm=True)
    try:
        for t in range(1, 3):
            r.step(t)
            p.assert_exact(r.compare(t + 1), "flat")
    finally:
        r.close()


# -----------------------------------------------------------------------------
# Algorithm 2 options and the Algorithm 2 (no bias correction) reading
# -----------------------------------------------------------------------------
@pytest.mark.parametrize("hp", [
    dict(g_max=0.7), dict(w_max=0.03), dict(wd_add=0.1), dict(dmult_max=0.02),
    dict(bias_correction=0), dict(lr_mul=0.0), dict(lr_add=0.0), dict(lr_mul=0.5, lr_add=0.05),
    dict(g_max=0.5, w_max=0.05, wd_add=0.01, dmult_max=0.1, rmax_neg=0.6, rmax_pos=0.5, tau=1e-3),
    # outside the certified fast path's conditions: the exact sequence runs throughout
    dict(eps=1e-10), dict(lr_mul=5.0), dict(beta2=0.9999999),
])
@pytest.mark.parametrize("name", ["gpt2_124m", "llama_1p5b"])
def test_algorithm2_options(hp, name):
    p = P()
    r = p.Run(W.SMALL[name], warm=True, hp=hp)
    try:
        for t in range(1, 4):
            r.step(t)
            p.assert_exact(r.compare(t + 1), f"{hp}")
    finally:
        r.close()


# -----------------------------------------------------------------------------
# Non-finite values propagate identically
# -----------------------------------------------------------------------------
@pytest.mark.parametrize("wd", ["bf16", "e4m3"])
def test_nan_and_inf_propagate_like_the_oracle(wd):
    p = P()
    wl = _edge_workload(wd, "f32", "bf16", "stochastic")
    mt = W.materialize(wl, "cpu", warm_state=True)
    big = max(range(len(mt.g)), key=lambda k: mt.g[k].numel())
    g = mt.g[big]
    g[::97] = float("nan")
    g[5::131] = float("inf")
    g[7::151] = -float("inf")
    if wd == "bf16":
        mt.w[big][11::173] = float("inf")
        mt.w[big][13::179] = float("nan")
    else:
        mt.w[big][11::173] = 0x7F  # NaN code
    mt.ve[big][17::191] = float("inf")
    r = p.Run(wl, mt=mt)
    try:
        for t in range(1, 3):
            r.step(t)
            p.assert_exact(r.compare(t + 1), "non-finite")
    finally:
        r.close()


# -----------------------------------------------------------------------------
# Many undecided elements: large learning rates (eta_m = 4 is the largest the
# certified path accepts) widen its error bound several times, so whole tiles
# send many more elements through the exact branch (for BF16 weights, one
# element at a time from the stage, with its random lane drawn again)
# -----------------------------------------------------------------------------
@pytest.mark.parametrize("wd", ["bf16", "e4m3"])
@pytest.mark.parametrize("gd,md", [("bf16", "bf16"), ("f32", "f32"), ("bf16", "f32")])
@pytest.mark.parametrize("rnd", ["nearest", "stochastic"])
def test_many_undecided_elements(wd, gd, md, rnd):
    p = P()
    wl = W.replace(W.SMALL["llama_7b"], weight_dtype=wd, grad_dtype=gd, moment_dtype=md, rounding=rnd,
                   name=f"undecided_{wd}")
    r = p.Run(wl, warm=True, hp=dict(lr_mul=4.0, lr_add=0.3))
    try:
        for t in range(1, 4):
            r.step(t)
            p.assert_exact(r.compare(t + 1), f"{wd}/{gd}/{md}/{rnd} step {t}")
    finally:
        r.close()


# -----------------------------------------------------------------------------
# E4M3 codes over their whole range (subnormal codes, values far below the
# smallest code after the update, saturation), where the certified path's
# fast encode is out of range and the exact branch must take over without
# touching its neighbours' bytes
# -----------------------------------------------------------------------------
@pytest.mark.parametrize("md", ["f32", "bf16"])
@pytest.mark.parametrize("rnd", ["nearest", "stochastic"])
def test_e4m3_codes_over_their_whole_range(md, rnd):
    import torch
    p = P()
    wl = W.replace(W.SMALL["llama_1p5b"], moment_dtype=md, rounding=rnd, name="e4m3_all_codes")
    mt = W.materialize(wl, "cpu", warm_state=True)
    gen = torch.Generator().manual_seed(5)
    finite = torch.tensor([c for c in range(256) if c & 0x7F != 0x7F], dtype=torch.uint8)
    for k, w in enumerate(mt.w):
        w.copy_(finite[torch.randint(0, finite.numel(), (w.numel(),), generator=gen)])
    r = p.Run(wl, mt=mt, hp=dict(lr_add=1e-2, lr_mul=0.05))
    try:
        for t in range(1, 5):
            r.step(t)
            res = r.compare(t + 1)
            assert res["contract_ok"]
            p.assert_exact(res, f"all codes {md}/{rnd} step {t}")
    finally:
        r.close()


# -----------------------------------------------------------------------------
# Weights far above 2^125 (up to near BF16's largest value): the certified
# path's third divisor max(|w|, tau) leaves the approximate division's range,
# where w + w u_m must still round to w as in the canonical sequence
# -----------------------------------------------------------------------------
@pytest.mark.parametrize("md", ["f32", "bf16"])
@pytest.mark.parametrize("rnd", ["nearest", "stochastic"])
def test_huge_weights(md, rnd):
    import torch
    p = P()
    wl = W.replace(W.SMALL["llama_7b"], moment_dtype=md, rounding=rnd, name="huge_weights")
    mt = W.materialize(wl, "cpu", warm_state=True)
    big = max(range(len(mt.w)), key=lambda k: mt.w[k].numel())
    w = mt.w[big]
    vals = torch.tensor([2.0 ** 125, -2.0 ** 126, 3.0e38, -3.3e38, 5.0e37, 2.0 ** 127], dtype=torch.float32)
    idx = torch.arange(0, w.numel(), 7)
    w[idx] = vals[torch.arange(idx.numel()) % vals.numel()].to(torch.bfloat16)
    r = p.Run(wl, mt=mt, hp=dict(lr_mul=4.0))
    try:
        for t in range(1, 4):
            r.step(t)
            p.assert_exact(r.compare(t + 1), f"huge weights {md}/{rnd} step {t}")
    finally:
        r.close()


# -----------------------------------------------------------------------------
# Launch shape and list structure do not change any bit
# -----------------------------------------------------------------------------
def test_grid_size_does_not_change_results():
    p = P()
    wl = W.SMALL["llama_7b"]
    runs = []
    for grid in (0, 1, 7, 333, 5000):
        r = p.Run(wl, warm=True)
        if grid:
            r.opt.set_grid(grid)
        for t in range(1, 3):
            r.step(t)
        runs.append(r)
    ref = runs[0]
    for r in runs:
        p.assert_exact(r.compare(3), "grid")
        for k in range(len(ref.dev["w"])):
            assert torch.equal(r.dev["w"][k], ref.dev["w"][k])
    for r in runs:
        r.close()


def test_split_at_multiple_of_8_is_bit_identical_on_gpu():
    p = P()
    from paper_2607_10611_gb300.optimizer import MPAdam
    wl = W.SMALL["gpt2_124m"]
    mt = W.materialize(wl, "cpu", warm_state=True)
    dev = {key: a for key, a in p.device_copy(mt).items() if key in ("w", "g", "m", "v", "ve")}
    # split every tensor with >= 16 elements at a multiple of 8 into two list entries
    cut = [((n // 2) // 8) * 8 for n in (t.numel() for t in dev["w"])]
    split = {key: [] for key in dev}
    clone = {key: [t.clone() for t in dev[key]] for key in dev}
    for k, c in enumerate(cut):
        for key in dev:
            t = clone[key][k]
            split[key] += [t[:c], t[c:]] if c > 0 else [t]
    kw = dict(weight_dtype=wl.weight_dtype, grad_dtype=wl.grad_dtype, moment_dtype=wl.moment_dtype,
              rounding=wl.rounding, seed=wl.seed)
    a = MPAdam(dev["w"], dev["m"], dev["v"], dev["ve"], **kw)
    b = MPAdam(split["w"], split["m"], split["v"], split["ve"], **kw)
    # the split list keeps every element's global index only if no padding is added:
    # offsets must coincide
    oa, ob = a.global_offsets(), b.global_offsets()
    j = 0
    for k, c in enumerate(cut):
        assert ob[j] == oa[k]
        j += 2 if c > 0 else 1
    for t in range(1, 4):
        a.step(dev["g"], t)
        b.step(split["g"], t)
    torch.cuda.synchronize()
    for key in ("w", "m", "v", "ve"):
        for k in range(len(dev["w"])):
            assert torch.equal(dev[key][k].view(torch.uint8), clone[key][k].view(torch.uint8)), key
    a.close(); b.close()


# -----------------------------------------------------------------------------
# Host-buffer entry point, random lanes, empty list
# -----------------------------------------------------------------------------
@pytest.mark.parametrize("layout", ["separate", "flat"])
def test_step_host_equals_device_step(layout):
    p = P()
    wl = W.SMALL["llama_1p5b"]
    r1 = p.Run(wl, warm=True, layout=layout)
    r2 = p.Run(wl, warm=True, layout=layout)
    try:
        if layout == "flat":
            hg_base = r2.mt.flat["g"].pin_memory()
            hw_base = torch.empty_like(r2.mt.flat["w"]).pin_memory()
            hg = [hg_base[o:o + t.numel()] for o, t in zip(r2.mt.offsets, r2.mt.g)]
            hw = [hw_base[o:o + t.numel()] for o, t in zip(r2.mt.offsets, r2.mt.w)]
        else:
            hg = [t.pin_memory() for t in r2.mt.g]
            hw = [torch.empty_like(t).pin_memory() for t in r2.mt.w]
        for t in range(1, 4):
            r1.opt.step(r1.dev["g"], t)
            r2.opt.step_host(hg, hw, t)
        torch.cuda.synchronize()
        for k in range(len(hw)):
            assert torch.equal(hw[k], r1.dev["w"][k].cpu())
            assert torch.equal(r2.dev["w"][k], r1.dev["w"][k])
            assert torch.equal(r2.dev["ve"][k], r1.dev["ve"][k])
    finally:
        r1.close(); r2.close()


@pytest.mark.parametrize("wd", ["bf16", "e4m3"])
def test_rng_lanes_match_oracle(wd):
    from paper_2607_10611_gb300 import _native as N
    rng = np.random.default_rng(3)
    for seed, step, first in [(0, 1, 0), (0xDEADBEEFCAFE, 77, 12345), (5, (1 << 33) + 9, (1 << 40) - 37)]:
        n = 20000
        out = torch.zeros(n, dtype=torch.int32, device="cuda")
        N.mpadam_rng_lanes(seed, step, N.DTYPE[wd], first, n, out.data_ptr())
        torch.cuda.synchronize()
        got = out.cpu().numpy().view(np.uint32)
        want = oracle.rng_lanes(seed, step, np.arange(first, first + n, dtype=np.uint64),
                                oracle.BF16 if wd == "bf16" else oracle.E4M3)
        np.testing.assert_array_equal(got, want)


def test_empty_list_and_zero_sized_tensors():
    from paper_2607_10611_gb300 import _native as N
    cfg = N.make_config()
    s = N.mpadam_create([], cfg)
    N.mpadam_step(s, [], 1)
    N.mpadam_destroy(s)
    z = torch.zeros(0, dtype=torch.bfloat16, device="cuda")
    zf = torch.zeros(0, dtype=torch.float32, device="cuda")
    s = N.mpadam_create([(0, 0, 0, 0, 0), (z.data_ptr(), zf.data_ptr(), zf.data_ptr(), zf.data_ptr(), 0)], cfg)
    N.mpadam_step(s, [0, 0], 1)
    torch.cuda.synchronize()
    N.mpadam_destroy(s)


def test_step_rejects_null_grads_on_gpu():
    from paper_2607_10611_gb300 import _native as N
    w = torch.zeros(16, dtype=torch.bfloat16, device="cuda")
    m = torch.zeros(16, device="cuda")
    s = N.mpadam_create([(w.data_ptr(), m.data_ptr(), m.data_ptr(), m.data_ptr(), 16)], N.make_config())
    with pytest.raises(N.MPAdamError):
        N.mpadam_step(s, [0], 1)
    with pytest.raises(N.MPAdamError):
        N.mpadam_step(s, [m.data_ptr() + 2], 1)   # misaligned fp32 gradient
    with pytest.raises(N.MPAdamError):
        N.mpadam_step(s, [m.data_ptr()], 0)        # step 0
    N.mpadam_destroy(s)


def test_step_host_with_huge_page_host_buffers():
    """mpadam_host_buffer_alloc buffers as the host side of the pipelined
    host-buffer step: same bits as the device step."""
    from paper_2607_10611_gb300.optimizer import HostBuffer
    p = P()
    wl = W.SMALL["llama_7b"]
    r1 = p.Run(wl, warm=True, layout="flat")
    r2 = p.Run(wl, warm=True, layout="flat")
    bg = HostBuffer(r2.mt.flat["g"].numel(), r2.mt.flat["g"].dtype)
    bw = HostBuffer(r2.mt.flat["w"].numel(), r2.mt.flat["w"].dtype)
    try:
        bg.tensor.copy_(r2.mt.flat["g"])
        hg = [bg.tensor[o:o + t.numel()] for o, t in zip(r2.mt.offsets, r2.mt.g)]
        hw = [bw.tensor[o:o + t.numel()] for o, t in zip(r2.mt.offsets, r2.mt.w)]
        for t in range(1, 4):
            r1.opt.step(r1.dev["g"], t)
            r2.opt.step_host(hg, hw, t)
        torch.cuda.synchronize()
        for k in range(len(hw)):
            assert torch.equal(hw[k], r1.dev["w"][k].cpu())
            assert torch.equal(r2.dev["w"][k], r1.dev["w"][k])
    finally:
        r1.close(); r2.close()
        bg.free(); bw.free()
