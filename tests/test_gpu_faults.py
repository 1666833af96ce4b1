"""Failure handling and resume, on the GPU, with faults made on the host:
an allocation the driver refuses (injected) makes each entry point return
MPADAM_EALLOC, release what it had, and work again afterwards; a step sequence
interrupted by a checkpoint (every state array copied out and into fresh
buffers) continues bit for bit."""
import pytest
import torch

import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2607_10611_gb300 import build
    build()


@pytest.fixture(autouse=True)
def _disarm():
    from paper_2607_10611_gb300 import _native as N
    yield
    N.mpadam_debug_fail_allocation(-1)


def P():
    import parity
    return parity


def test_create_reports_every_refused_allocation_and_recovers():
    from paper_2607_10611_gb300 import _native as N
    p = P()
    wl = W.SMALL["llama_1p5b_nvfp4"]
    failures = 0
    for after in range(12):
        N.mpadam_debug_fail_allocation(after)
        try:
            r = p.Run(wl, warm=True)
        except N.MPAdamError as e:
            assert e.status == N.MPADAM_EALLOC, e
            failures += 1
            continue
        finally:
            N.mpadam_debug_fail_allocation(-1)
        r.close()
    assert failures >= 5            # descriptor, grad, aux, error-word, pinned tables and the CTA tables
    r = p.Run(wl, warm=True)        # nothing left behind: a full run still matches the oracle
    try:
        for t in (1, 2):
            r.step(t)
            p.assert_exact(r.compare(t + 1), f"after injected failures, step {t}")
    finally:
        r.close()


def test_host_buffer_step_staging_failure_then_success():
    from paper_2607_10611_gb300 import _native as N
    p = P()
    wl = W.SMALL["llama_7b"]
    r1, r2 = p.Run(wl, warm=True, layout="flat"), p.Run(wl, warm=True, layout="flat")
    try:
        hg = [t.pin_memory() for t in r2.mt.g]
        hw = [torch.empty_like(t).pin_memory() for t in r2.mt.w]
        N.mpadam_debug_fail_allocation(0)          # the gradient staging buffer
        with pytest.raises(N.MPAdamError) as ei:
            r2.opt.step_host(hg, hw, 1)
        assert ei.value.status == N.MPADAM_EALLOC
        N.mpadam_debug_fail_allocation(-1)
        for t in (1, 2):
            r1.opt.step(r1.dev["g"], t)
            r2.opt.step_host(hg, hw, t)
        torch.cuda.synchronize()
        for k in range(len(hw)):
            assert torch.equal(r2.dev["w"][k], r1.dev["w"][k])
            assert torch.equal(hw[k], r1.dev["w"][k].cpu())
    finally:
        r1.close(); r2.close()


def test_toy_create_failure_then_success():
    from paper_2607_10611_gb300 import _native as N
    from paper_2607_10611_gb300.toy import ToyDiagnostic
    p = W.toy_problem("sign_flip", n=64)
    w, ws = p.w0.to("cuda"), p.wstar.to("cuda")
    for after in range(4):
        N.mpadam_debug_fail_allocation(after)
        with pytest.raises(N.MPAdamError):
            ToyDiagnostic(w, ws, mode="combined", batch=64, lr_add=1.0, lr_mul=1.0)
    N.mpadam_debug_fail_allocation(-1)
    d = ToyDiagnostic(w, ws, mode="combined", batch=64, lr_add=1.0, lr_mul=1.0)
    d.run(1, 10)
    torch.cuda.synchronize()
    d.close()


@pytest.mark.parametrize("name", ["llama_7b", "llama_1p5b", "llama_1p5b_mixed", "llama_1p5b_nvfp4"])
def test_checkpoint_and_resume_is_bit_exact(name):
    """2k steps in one go equal k steps, a checkpoint (weights, moments, block
    scales and the E4M3 scale rings copied to host memory and back into fresh
    device buffers with a fresh optimizer state), then k more steps."""
    p = P()
    wl = W.SMALL[name]
    k = 3
    ref = p.Run(wl, warm=True)
    part = p.Run(wl, warm=True)
    try:
        for t in range(1, 2 * k + 1):
            ref.opt.step(ref.dev["g"], t)
        for t in range(1, k + 1):
            part.opt.step(part.dev["g"], t)
        torch.cuda.synchronize()
        keys = ("w", "m", "v", "ve", "bscale")
        saved = {key: [None if x is None else x.cpu() for x in part.dev[key]] for key in keys}
        rings = None
        if part.opt.fp8_exp_ring is not None:
            rings = (part.opt.fp8_exp_ring.cpu(), part.opt.fp8_amax_ring.cpu())
        part.close()
        # restore into new buffers and a new state
        res = p.Run(wl, warm=True)
        for key in keys:
            for dst, src in zip(res.dev[key], saved[key]):
                if dst is not None:
                    dst.copy_(src)
        if rings is not None:
            res.opt.fp8_exp_ring.copy_(rings[0])
            res.opt.fp8_amax_ring.copy_(rings[1])
        for t in range(k + 1, 2 * k + 1):
            res.opt.step(res.dev["g"], t)
        torch.cuda.synchronize()
        for key in keys:
            for a, b in zip(res.dev[key], ref.dev[key]):
                if a is not None:
                    assert torch.equal(a.view(torch.uint8), b.view(torch.uint8)), key
        if rings is not None:
            assert torch.equal(res.opt.fp8_exp_ring, ref.opt.fp8_exp_ring)
            assert torch.equal(res.opt.fp8_amax_ring, ref.opt.fp8_amax_ring)
        res.close()
    finally:
        ref.close()
