"""mpadam_step_noalloc: the entry point for callers that must not call
cudaMalloc (a runtime whose device memory all belongs to its own caching
allocator or memory pool, or a service that fixes its device-memory budget at
start-up).  It keeps its tables in one device array built into the library
instead of allocating, so it must give exactly what mpadam_step gives on the
same inputs -- checked here bit for bit, the tolerance of every other parity
test, over two calls in a row that reuse that shared array.  After the calls,
mpadam_noalloc_status must report that no bounded wait inside the step kernel
gave up (that word lives in the same array).

Lists covered: more tensors than one table-fill launch carries (384), the
E4M3 and BF16-moment formats, empty tensors passed with NULL pointers, and
exactly the 8192-tensor limit.  The per-CTA table's own limit (4096 CTAs) is
not reachable here: the step kernel runs one CTA per SM.

The file name makes pytest collect it last, so a failure here leaves every
other test already run; it also passes alone in a fresh process.
"""
import pytest
import torch

import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def N():
    from paper_2607_10611_gb300 import _native, build
    build()
    return _native


def _with_empty_tensors():
    """A ragged list with zero-length tensors at the start, the middle and the end."""
    specs = W.ragged_specs(40, 14, 5)
    empty = W.TensorSpec("empty", 0, "flat")
    specs = (empty,) + specs[:20] + (empty, empty) + specs[20:] + (empty,)
    return W.replace(W.SMALL["ragged_20k"], specs=specs, name="ragged_with_empty")


def _lists():
    ragged = W.replace(W.SMALL["ragged_20k"], specs=W.ragged_specs(1000, 10, 3), name="ragged_1000")
    limit = W.replace(W.SMALL["ragged_20k"], specs=W.ragged_specs(8192, 6, 9), name="ragged_8192")
    return [ragged, W.SMALL["llama_1p5b"], W.SMALL["llama_7b"], _with_empty_tensors(), limit]


def _device(mt):
    return {key: [t.to("cuda") for t in getattr(mt, key)] for key in ("w", "g", "m", "v", "ve")}


@pytest.mark.parametrize("wl", _lists(), ids=lambda w: w.name)
def test_noalloc_matches_mpadam_step_on_two_calls(N, wl):
    from paper_2607_10611_gb300.optimizer import MPAdam
    mt = W.materialize(wl, "cpu", warm_state=True)
    a, b = _device(mt), _device(mt)
    ref = MPAdam(a["w"], a["m"], a["v"], a["ve"], weight_dtype=wl.weight_dtype,
                 grad_dtype=wl.grad_dtype, moment_dtype=wl.moment_dtype, rounding=wl.rounding,
                 seed=wl.seed, fp8_exp=mt.fp8_exp)
    cfg = N.make_config(weight_dtype=wl.weight_dtype, grad_dtype=wl.grad_dtype,
                        moment_dtype=wl.moment_dtype, rounding=wl.rounding, seed=wl.seed)
    exp_ring = amax_ring = None
    if wl.weight_dtype == "e4m3":  # the caller's rings, seeded like the reference's
        torch.cuda.synchronize()
        exp_ring = ref.fp8_exp_ring.clone()
        amax_ring = ref.fp8_amax_ring.clone()

    def ptr(t):  # empty tensors go in with NULL pointers
        return t.data_ptr() if t.numel() else 0

    tensors = [(ptr(w), ptr(m), ptr(v), ptr(ve), w.numel())
               for w, m, v, ve in zip(b["w"], b["m"], b["v"], b["ve"])]
    grads = [ptr(g) for g in b["g"]]
    stream = torch.cuda.current_stream().cuda_stream
    for t in (1, 2):
        ref.step(a["g"], t)
        N.mpadam_step_noalloc(tensors, grads, cfg, t,
                              exp_ring.data_ptr() if exp_ring is not None else 0,
                              amax_ring.data_ptr() if amax_ring is not None else 0, stream)
        torch.cuda.synchronize()
        for key in ("w", "m", "v", "ve"):
            for x, y in zip(a[key], b[key]):
                assert torch.equal(x.view(torch.uint8), y.view(torch.uint8)), (wl.name, t, key)
        if exp_ring is not None:
            assert torch.equal(exp_ring, ref.fp8_exp_ring)
            assert torch.equal(amax_ring, ref.fp8_amax_ring)
    assert N.mpadam_noalloc_status(stream) == 0, "a bounded wait in the allocation-free step gave up"
    assert ref.device_status() == 0
    ref.close()


def test_noalloc_rejects_lists_beyond_its_limit(N):
    cfg = N.make_config()
    w = torch.zeros(8, dtype=torch.bfloat16, device="cuda")
    m = torch.zeros(8, device="cuda")
    t = (w.data_ptr(), m.data_ptr(), m.data_ptr(), m.data_ptr(), 8)
    with pytest.raises(N.MPAdamError) as ei:
        N.mpadam_step_noalloc([t] * 8193, [m.data_ptr()] * 8193, cfg, 1)
    assert ei.value.status == N.MPADAM_EINVAL and "8192" in str(ei.value)
    with pytest.raises(N.MPAdamError) as ei:  # no place for the code
        N._check(N.lib().mpadam_noalloc_status(None, None))
    assert ei.value.status == N.MPADAM_EINVAL
