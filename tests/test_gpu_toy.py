"""GPU parity of the BF16-stored matrix-fitting diagnostic (the toy
diagnostic of Sec. 5.1 and its appendix): weights and per-step minibatch
losses bit for bit against the oracle, in all five regimes and all three
update rules, at the paper's size (n = 4096, W of 16.8M entries) and on a
small problem where entries are sampled many times."""
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


LR = {"additive": dict(lr_add=1024.0), "multiplicative": dict(lr_mul=1024.0),
      "combined": dict(lr_add=1024.0, lr_mul=1024.0)}


def _compare(regime, mode, n, batch, steps, lr_scale=1.0):
    from paper_2607_10611_gb300.toy import ToyDiagnostic
    p = W.toy_problem(regime, n=n, seed=5)
    lr = {k: v * lr_scale for k, v in LR[mode].items()}
    dev_w = p.w0.to("cuda")
    dev_ws = p.wstar.to("cuda")
    d = ToyDiagnostic(dev_w, dev_ws, mode=mode, batch=batch, c_lo=p.c_lo, c_hi=p.c_hi, split=p.split, seed=11, **lr)
    losses = torch.zeros(steps, dtype=torch.float64, device="cuda")
    for t in range(1, steps + 1):
        d.step(t, loss_out=losses[t - 1:t])
    torch.cuda.synchronize()
    hw = W.to_numpy_bits(p.w0)
    hs = p.wstar.numpy()
    cfg = oracle.toy_config(mode, batch=batch, c_lo=p.c_lo, c_hi=p.c_hi, split=p.split, seed=11, **lr)
    want = np.array([oracle.toy_step(cfg, hw, hs, t) for t in range(1, steps + 1)])
    got_w = W.to_numpy_bits(dev_w)
    bad = int((got_w != hw).sum())
    assert bad == 0, f"{regime}/{mode}: {bad} weights differ"
    np.testing.assert_array_equal(losses.cpu().numpy().view(np.uint64), want.view(np.uint64))
    d.close()
    return want


@pytest.mark.parametrize("mode", ["additive", "multiplicative", "combined"])
@pytest.mark.parametrize("regime", W.TOY_REGIMES)
def test_toy_full_size_bit_exact(regime, mode):
    _compare(regime, mode, W.TOY_N, 65536, 6)


@pytest.mark.parametrize("mode", ["additive", "multiplicative", "combined"])
@pytest.mark.parametrize("regime", W.TOY_REGIMES)
def test_toy_small_many_repeats_bit_exact(regime, mode):
    """n = 64 (4096 entries), B = 64: every entry is hit about once every 64
    steps and repeated hits within a step are common."""
    losses = _compare(regime, mode, 64, 64, 200, lr_scale=1.0 / 1024.0)
    assert np.all(np.isfinite(losses))


def test_toy_rejects_bad_arguments():
    from paper_2607_10611_gb300 import _native as N
    ok = dict(mode=2, split=0, batch=64, reserved=0, lr_add=1.0, lr_mul=1.0, rmax=0.75, tau=1e-8, c_lo=1.0,
              c_hi=1.0, seed=0)
    for n, over in [(100, {}), (64, {"batch": 48}), (64, {"batch": 32, "split": 1}), (64, {"mode": 3}),
                    (64, {"tau": 0.0}), (64, {"lr_add": -1.0}), (64, {"reserved": 1})]:
        cfg = N.mpadam_toy_config(**{**ok, **over})
        with pytest.raises(N.MPAdamError):
            N.mpadam_toy_create(n, cfg)


@pytest.mark.parametrize("regime", ["sign_flip", "mixed"])
def test_toy_run_graph_replays_equal_single_steps(regime):
    """mpadam_toy_run (CUDA-graph replays of 64 steps, a plain remainder,
    the step number in device memory) gives the bits of step-by-step calls,
    also when called again and with new pointers (a new capture)."""
    from paper_2607_10611_gb300.toy import ToyDiagnostic
    p = W.toy_problem(regime, n=256, seed=3)
    kw = dict(mode="combined", batch=1024, c_lo=p.c_lo, c_hi=p.c_hi, split=p.split, seed=2,
              lr_add=48.0, lr_mul=48.0)
    ws = p.wstar.to("cuda")
    w1, w2 = p.w0.to("cuda"), p.w0.to("cuda")
    d1, d2 = ToyDiagnostic(w1, ws, **kw), ToyDiagnostic(w2, ws, **kw)
    steps = 2 * 64 + 5
    l1 = torch.zeros(steps, dtype=torch.float64, device="cuda")
    for t in range(1, steps + 1):
        d1.step(t, loss_out=l1[t - 1:t])
    l2 = torch.zeros(steps, dtype=torch.float64, device="cuda")
    d2.run(1, 70, l2[:70])
    d2.run(71, steps - 70, l2[70:])       # new losses pointer: a new capture
    torch.cuda.synchronize()
    assert torch.equal(w1, w2)
    assert torch.equal(l1, l2)
    d1.close(); d2.close()
