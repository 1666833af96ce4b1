"""Pins of the oracle's BF16-stored matrix-fitting diagnostic (the toy
diagnostic of Sec. 5.1 and its appendix): the tree-ordered mean, the
gradient of c (mean r^2)^2 with repeated samples, the sampling, and the
regime behaviours the paper reports (multiplicative steps keep signs and
cannot leave zero; additive steps stall at large magnitudes)."""
import numpy as np
import pytest

import oracle
import workloads as W

F = np.float32


def test_tree_sum_is_the_adjacent_pair_tree():
    # tree: (1e16 + 1) + (-1e16 + 1) = 1e16 + -1e16 = 0 ; left to right gives 1
    assert oracle.tree_sum([1e16, 1.0, -1e16, 1.0]) == 0.0
    rng = np.random.default_rng(0)
    x = rng.standard_normal(1024)
    from fractions import Fraction
    exact = sum(Fraction(v) for v in x)
    assert abs(Fraction(oracle.tree_sum(x)) - exact) <= 1024 * 2.0 ** -52 * sum(abs(Fraction(v)) for v in x)


def _lanes_idx(seed, t, B, rng_range, split, n):
    lanes = oracle.rng_lanes(seed, t, np.arange(B, dtype=np.uint64), oracle.E4M3).astype(np.int64)
    idx = lanes & (rng_range - 1)
    if split:
        idx[B // 2:] += n // 2
    return idx


@pytest.mark.parametrize("split", [False, True])
def test_gradient_closed_form_with_repeated_samples(split):
    """w = 1/2, w* = 0 everywhere: every residual is 1/2, M = 1/4, and an
    entry hit k times gets g = k * 4 c M (1/2) / B_h; with c = 1, B = 64
    (B_h = 64 or 32) and eta_a = 1 the additive step lands exactly on
    1/2 - k / 128 (or k / 64), BF16-representable."""
    n, B = 256, 64
    w = np.full(n, oracle.bf16_rne([0.5])[0], np.uint16)
    ws = np.zeros(n, F)
    cfg = oracle.toy_config("additive", lr_add=1.0, batch=B, c_lo=1.0, split=split, seed=3)
    loss = oracle.toy_step(cfg, w, ws, 5)
    assert loss == (2.0 if split else 1.0) * (1.0 / 16.0)      # sum over halves of c M^2, M = 1/4
    idx = _lanes_idx(3, 5, B, n // 2 if split else n, split, n)
    k = np.bincount(idx, minlength=n)
    step = 1.0 / (64.0 if split else 128.0)
    want = oracle.bf16_rne((0.5 - k * step).astype(F))
    np.testing.assert_array_equal(w, want)
    assert (k > 1).any()          # the batch has repeated entries


def test_multiplicative_step_scales_by_ln2():
    """Same setting, multiplicative: u_m = -eta_m ln2 g (w > 0), so w' =
    w (1 - eta_m ln2 g); with eta_m = 1 / ln2 the result is 1/2 (1 - k/128)
    to within one BF16 rounding."""
    n, B = 256, 64
    w = np.full(n, oracle.bf16_rne([0.5])[0], np.uint16)
    cfg = oracle.toy_config("multiplicative", lr_mul=1.0 / np.log(2.0), batch=B, seed=3)
    oracle.toy_step(cfg, w, np.zeros(n, F), 5)
    k = np.bincount(_lanes_idx(3, 5, B, n, False, n), minlength=n)
    got = oracle.bf16_decode(w).astype(np.float64)
    want = 0.5 * (1.0 - k / 128.0)
    assert np.all(np.abs(got - want) <= 2.0 ** -9 * np.maximum(want, 1e-30))


def test_batch_loss_is_c_mean_square_squared():
    rng = np.random.default_rng(1)
    n, B = 1024, 128
    w = oracle.bf16_rne(rng.standard_normal(n).astype(F))
    ws = rng.standard_normal(n).astype(F)
    cfg = oracle.toy_config("combined", batch=B, c_lo=3.0, seed=8)
    loss = oracle.toy_step(cfg, w.copy(), ws, 2)
    idx = _lanes_idx(8, 2, B, n, False, n)
    r = (oracle.bf16_decode(w)[idx] - ws[idx]).astype(F).astype(np.float64)
    assert loss == pytest.approx(3.0 * np.mean(r * r) ** 2, rel=1e-12)


def _run(regime, mode, steps, n=64, B=64, **lr):
    p = W.toy_problem(regime, n=n, seed=2)
    w = W.to_numpy_bits(p.w0)
    ws = p.wstar.numpy()
    cfg = oracle.toy_config(mode, batch=B, c_lo=p.c_lo, c_hi=p.c_hi, split=p.split, seed=4, **lr)
    losses = [oracle.toy_step(cfg, w, ws, t) for t in range(1, steps + 1)]
    return w, ws, losses, p


def test_multiplicative_keeps_signs_in_the_sign_flip_regime():
    w, ws, losses, p = _run("sign_flip", "multiplicative", 300, lr_mul=1e3)
    w0 = oracle.bf16_decode(W.to_numpy_bits(p.w0))
    got = oracle.bf16_decode(w)
    assert np.all((got == 0) | (np.sign(got) == np.sign(w0)))
    assert np.all(np.sign(got) != np.sign(ws))     # never reaches the other side


def test_multiplicative_cannot_leave_zero():
    w, ws, losses, p = _run("zero_revival", "multiplicative", 100, lr_mul=1e3)
    assert np.all(oracle.bf16_decode(w) == 0)
    assert losses[-1] == losses[0]


def test_additive_stalls_at_large_weights_below_half_an_ulp():
    """BF16 spacing at 100 is 0.5: steps below 0.25 round away (Sec. 5.1).
    With B = 64 here, eta_a = 0.01 keeps every additive step (repeated hits
    included) below 0.25, so no weight moves, while the combined step,
    whose multiplicative branch is relative, moves most of them."""
    w, ws, losses, p = _run("large", "additive", 100, lr_add=0.01)
    assert np.all(oracle.bf16_decode(w) == 100.0)
    w, ws, losses, p = _run("large", "combined", 100, lr_add=0.01, lr_mul=0.01)
    assert np.mean(oracle.bf16_decode(w) != 100.0) > 0.5


@pytest.mark.parametrize("regime", W.TOY_REGIMES)
def test_combined_makes_progress_in_every_regime(regime):
    """One shared learning rate (eta_a = eta_m) for all five regimes, as the
    paper's main diagnostic figure uses (scaled here to B = 64)."""
    w, ws, losses, p = _run(regime, "combined", 400, lr_add=1.0, lr_mul=1.0)
    assert np.mean(losses[-20:]) < 0.5 * np.mean(losses[:5])
