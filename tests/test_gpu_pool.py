"""GPU parity with the tail pool on: the last part of every CTA's run of
tiles goes to a pool that the CTAs finishing first claim chunk by chunk.
Which CTA steps which tile must not change a single stored bit, nor the
E4M3 scale rings: every format, pool shares from all-static to all-pooled,
chunk lengths, and grids with more CTAs than tiles."""
import pytest
import torch

import workloads as W

pytestmark = pytest.mark.gpu

# (static share in 1/1024, chunk tiles, grid; 0 = default)
SETTINGS = [(0, 1, 0), (512, 3, 0), (900, 2, 7), (0, 5, 333), (768, 1, 1), (1024, 4, 0)]


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2607_10611_gb300 import build
    build()


def P():
    import parity
    return parity


@pytest.mark.parametrize("name", ["llama_7b", "llama_1p5b", "llama_1p5b_mixed", "llama_1p5b_nvfp4", "ragged_20k"])
@pytest.mark.parametrize("q,chunk,grid", SETTINGS)
def test_tail_pool_keeps_every_bit(name, q, chunk, grid):
    p = P()
    r = p.Run(W.SMALL[name], warm=True)
    try:
        if grid:
            r.opt.set_grid(grid)
        r.opt.set_tail_pool(q, chunk)
        for t in range(1, 4):
            r.step(t)
            res = r.compare(t + 1)
            p.assert_exact(res, f"{name} pool q={q} chunk={chunk} grid={grid} step {t}")
    finally:
        r.close()


def test_tail_pool_on_a_list_of_many_tiles_matches_static_runs():
    """Hundreds of pool chunks claimed concurrently by all CTAs: the result
    equals the static split's, bit for bit, over several steps."""
    from paper_2607_10611_gb300.optimizer import MPAdam
    wl = W.replace(W.SMALL["ragged_20k"], name="ragged_more")
    specs = tuple(W.TensorSpec(f"t{i}", 3840 * (1 + (7 * i) % 23) + (i % 5), "matrix") for i in range(300))
    wl = W.replace(wl, specs=specs)
    outs = []
    for q, chunk in ((1024, 4), (256, 2), (0, 1)):
        mt = W.materialize(wl, "cuda", layout="flat")
        opt = MPAdam(mt.w, mt.m, mt.v, mt.ve, weight_dtype=wl.weight_dtype, grad_dtype=wl.grad_dtype,
                     moment_dtype=wl.moment_dtype, rounding=wl.rounding, seed=3)
        opt.set_tail_pool(q, chunk)
        for t in range(1, 4):
            opt.step(mt.g, t)
        torch.cuda.synchronize()
        assert opt.device_status() == 0
        outs.append([x.clone() for x in (mt.flat["w"], mt.flat["m"], mt.flat["v"], mt.flat["ve"])])
        opt.close()
    for o in outs[1:]:
        for a, b in zip(outs[0], o):
            assert torch.equal(a.view(torch.int16) if a.dtype == torch.bfloat16 else a.view(torch.int32),
                               b.view(torch.int16) if b.dtype == torch.bfloat16 else b.view(torch.int32))


def test_set_tail_pool_rejects_bad_values():
    from paper_2607_10611_gb300 import _native as N
    r = P().Run(W.SMALL["llama_7b"])
    try:
        for q, chunk in ((-1, 4), (1025, 4), (512, 0), (512, (1 << 20) + 1)):
            with pytest.raises(N.MPAdamError) as ei:
                r.opt.set_tail_pool(q, chunk)
            assert ei.value.status == N.MPADAM_EINVAL
    finally:
        r.close()
