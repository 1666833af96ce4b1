"""GPU parity on short lists: a launch of at most four tensors (a flat
parameter buffer, a short list) carries its descriptors, aux entries and
gradient pointers in the kernel parameters, and each CTA finds its first
tensor by scanning them instead of reading the host-computed table.  Every
stored bit must still match the oracle: each weight format, one to five
tensors (five uses the tables), empty tensors at either end and in the
middle, tensors shorter than a tile, last tiles of whole warps only, grids
with more CTAs than tiles, and the tail pool on and off."""
import pytest

import workloads as W

pytestmark = pytest.mark.gpu

LISTS = {
    "one": (70001,),
    "two_empty_ends": (0, 9000, 5),
    "four": (3, 0, 20000, 7700),
    "five_tables": (3841, 1, 0, 12000, 64),
    # last tiles made of whole warps only (256 elements each): they take the
    # whole-tile path with no element-wise warp
    "warp_tails": (4096, 8448, 512),
}


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2607_10611_gb300 import build
    build()


def P():
    import parity
    return parity


def _workload(sizes, fmt, rnd):
    specs = tuple(W.TensorSpec(f"t{i}", n, "matrix") for i, n in enumerate(sizes))
    return W.Workload(name=f"short_{fmt}", specs=specs, weight_dtype=fmt, grad_dtype="bf16", moment_dtype="f32",
                      rounding=rnd, steps=3, seed=23, zero_frac=0.05, grad=("normal_logu", 1e-6, 1e-2),
                      compute_copy=fmt in ("e4m3_b32", "nvfp4"),
                      format_list=tuple([fmt] * len(sizes)) if fmt in ("e4m3_b32", "nvfp4") else ())


@pytest.mark.parametrize("fmt", ["bf16", "e4m3", "e4m3_b32", "nvfp4"])
@pytest.mark.parametrize("name", list(LISTS))
@pytest.mark.parametrize("grid,pool", [(0, None), (1, (1024, 4)), (7, (0, 1)), (64, None)])
@pytest.mark.parametrize("rnd", ["nearest", "stochastic"])
def test_short_lists_bit_exact(fmt, name, grid, pool, rnd):
    p = P()
    r = p.Run(_workload(LISTS[name], fmt, rnd), warm=True)
    try:
        if grid:
            r.opt.set_grid(grid)
        if pool:
            r.opt.set_tail_pool(*pool)
        for t in range(1, 4):
            r.step(t)
            p.assert_exact(r.compare(t + 1), f"{fmt} {name} grid={grid} pool={pool} step {t}")
    finally:
        r.close()
