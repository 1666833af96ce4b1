"""Pins of the oracle's M+Adam update against what the paper and mathematics fix.

P1  eta_m = 0 reduces M+Adam to Adam / AdamW (Sec. 3 eq. for AdamW vs the
    additive branch of Algorithm 1): pinned to torch.optim.Adam / AdamW.
P2  eta_a = 0 is the purely multiplicative update: sign-preserving and
    zero-absorbing, relative change bounded by the clip (Table 1; Fig. 1).
P3  zero weights: g_e = 0, so the update is the additive branch alone and
    nu_e only decays (Table 1 "can escape zero").
P4  closed forms of the first two steps from a zero state, derived by hand
    from Algorithm 1's definitions and evaluated in binary64.
P5  large-|w| stall of the additive branch under BF16 storage and its cure by
    the multiplicative branch (Sec. 1, Fig. 1, Table 1).
P8  the log2/exp2 step cap of Algorithm 2 equals a clamp of u_m.
P9  splitting a tensor at a multiple of 8 does not change any stored bit.
P10 descent on a quadratic (Theorem 4.1, idealised).
P11 resume: k + k steps equal 2k steps bit for bit.
"""
import copy
import math

import numpy as np
import pytest
import torch

import oracle
from oracle import BF16, E4M3, F32

F = np.float32
ULP = 2.0 ** -23


def _rand(n, seed, scale=1.0):
    return (np.random.default_rng(seed).standard_normal(n) * scale).astype(F)


# ----------------------------------------------------------------------------
# P1: Adam / AdamW limit
# ----------------------------------------------------------------------------
@pytest.mark.parametrize("wd", [0.0, 0.1])
def test_p1_adam_limit_matches_torch(wd):
    n, steps, lr = 4096, 40, 1e-3
    w0 = _rand(n, 0, 0.02)
    hp = oracle.hparams(lr_add=lr, lr_mul=0.0, beta1=0.9, beta2=0.999, eps=1e-8, wd_add=wd)
    w = w0.copy(); m = np.zeros(n, F); v = np.zeros(n, F); ve = np.zeros(n, F)
    p = torch.nn.Parameter(torch.from_numpy(w0.copy()))
    opt = (torch.optim.AdamW([p], lr=lr, betas=(0.9, 0.999), eps=1e-8, weight_decay=wd, foreach=False)
           if wd else torch.optim.Adam([p], lr=lr, betas=(0.9, 0.999), eps=1e-8, foreach=False))
    for t in range(1, steps + 1):
        g = _rand(n, 100 + t, 1e-3)
        oracle.step_elements(hp, t, F32, F32, F32, w, g.copy(), m, v, ve)
        p.grad = torch.from_numpy(g.copy())
        opt.step()
    ref = p.detach().numpy()
    # differing rounding orders: a few binary32 ulps of the weight per step
    tol = steps * 4 * ULP * np.maximum(np.abs(ref), 1e-3) + 1e-9
    assert np.all(np.abs(w - ref) <= tol)
    st = opt.state[p]
    # moments: EMA sums cancel, so bound the error by the summands' scale
    np.testing.assert_allclose(m, st["exp_avg"].numpy(), rtol=1e-5, atol=1e-6 * 1e-3)
    np.testing.assert_allclose(v, st["exp_avg_sq"].numpy(), rtol=1e-5, atol=1e-6 * 1e-6)


def test_p1_eta_m_zero_leaves_w_plus_ua_exactly():
    n = 2048
    w = _rand(n, 1, 0.05); g = _rand(n, 2, 1e-3)
    m = _rand(n, 3, 1e-4); v = (_rand(n, 4, 1e-3) ** 2).astype(F); ve = (_rand(n, 5, 1e-5) ** 2).astype(F)
    hp0 = oracle.hparams(lr_mul=0.0)
    wn, m1, v1, _ = oracle.update_elements(hp0, 7, w, g, m, v, ve)
    # u_a rebuilt from the moments with the Adam formula in binary64
    b1, b2 = float(F(0.9)), float(F(0.999))
    ua = -float(F(1e-3)) * (m1.astype(np.float64) / (1 - b1 ** 7)) / (
        np.sqrt(v1.astype(np.float64) / (1 - b2 ** 7)) + float(F(1e-8)))
    err = np.abs(wn.astype(np.float64) - (w.astype(np.float64) + ua))
    assert np.all(err <= 4 * ULP * (np.abs(w) + np.abs(ua)) + 1e-30)


# ----------------------------------------------------------------------------
# P2: purely multiplicative limit
# ----------------------------------------------------------------------------
def test_p2_multiplicative_only_preserves_sign_and_zero():
    n = 20000
    rng = np.random.default_rng(7)
    w = (rng.standard_normal(n) * 10.0 ** rng.uniform(-6, 2, n)).astype(F)
    w[::17] = 0.0
    w[1::53] = -0.0
    g = (rng.standard_normal(n) * 10.0 ** rng.uniform(-6, 0, n)).astype(F)
    m = np.zeros(n, F); v = np.zeros(n, F)
    ve = (rng.random(n) * 1e-6).astype(F)
    hp = oracle.hparams(lr_add=0.0, lr_mul=0.05)
    for t in (1, 3, 50):
        wn, _, _, _ = oracle.update_elements(hp, t, w, g, m, v, ve)
        z = w == 0
        assert np.all(wn[z] == 0)                        # zero-absorbing
        nz = ~z
        assert np.all(np.sign(wn[nz]) == np.sign(w[nz]))  # sign-preserving
        rel = wn[nz].astype(np.float64) / w[nz] - 1
        assert np.all(np.abs(rel) <= 0.75 * (1 + 4 * ULP))
        assert np.any(np.abs(rel) > 0.5)                 # the clip is reached somewhere


# ----------------------------------------------------------------------------
# P3: zero weights
# ----------------------------------------------------------------------------
def test_p3_zero_weights_take_the_additive_step_only():
    n = 1000
    w = np.zeros(n, F); g = _rand(n, 11, 1e-2)
    m = _rand(n, 12, 1e-3); v = (_rand(n, 13, 1e-2) ** 2).astype(F)
    ve = (np.abs(_rand(n, 14, 1e-4))).astype(F)
    a = oracle.update_elements(oracle.hparams(lr_mul=0.3), 5, w, g, m, v, ve)
    b = oracle.update_elements(oracle.hparams(lr_mul=0.0), 5, w, g, m, v, ve)
    np.testing.assert_array_equal(a[0].view(np.uint32), b[0].view(np.uint32))
    np.testing.assert_array_equal(a[3], (F(0.999) * ve).astype(F))   # nu_e only decays
    assert np.all(a[0] != 0)                                          # escapes zero


# ----------------------------------------------------------------------------
# P4: closed forms of the first steps
# ----------------------------------------------------------------------------
W_HAND = np.array([1.0, -2.0, 0.5, 0.0, 256.0, 1e-9, -0.03, 3e-3, 1.0, -1.0], F)
G_HAND = np.array([0.5, -0.5, 1e-3, -1e-3, 0.5, 1e-3, 2e-2, -1e-3, 1e-8, 3e-9], F)


def _closed_form_t1(w, g, lr_a, lr_m, b1, b2, eps, tau, gmax=math.inf):
    """Step 1 from mu = nu = nu_e = 0 with bias correction: mu-hat = g,
    sqrt(nu-hat) = |g|, sqrt(nu_e-hat) = |g_e|; so u_a = -lr_a g / (|g| + eps),
    n = g_e / (|g_e| + eps), u_m = clip(-lr_m n / max(|w|, tau))."""
    w = w.astype(np.float64); g = g.astype(np.float64)
    ge = math.log(2.0) * w * g
    ua = -lr_a * g / (np.abs(g) + eps)
    n = np.clip(ge / (np.abs(ge) + eps), -gmax, gmax)
    um = np.clip(-lr_m * n / np.maximum(np.abs(w), tau), -0.75, 0.75)
    wn = w + w * um + ua
    return wn, (1 - b1) * g, (1 - b2) * g * g, (1 - b2) * ge * ge, ua, w * um


@pytest.mark.parametrize("lr_a,lr_m,gmax", [(1e-3, 1e-3, math.inf), (1e-2, 0.3, math.inf),
                                             (1e-3, 2.0, math.inf), (1e-3, 1e-2, 0.5)])
def test_p4_first_step_closed_form(lr_a, lr_m, gmax):
    b1, b2, eps, tau = F(0.9), F(0.999), F(1e-8), F(1e-8)
    hp = oracle.hparams(lr_add=lr_a, lr_mul=lr_m, g_max=gmax)
    z = np.zeros_like(W_HAND)
    wn, m1, v1, ve1 = oracle.update_elements(hp, 1, W_HAND, G_HAND, z, z, z)
    ref_w, ref_m, ref_v, ref_ve, ua, mul = _closed_form_t1(
        W_HAND, G_HAND, F(lr_a), F(lr_m), float(b1), float(b2), float(eps), float(tau), gmax)
    scale = np.abs(W_HAND) + np.abs(ua) + np.abs(mul)
    assert np.all(np.abs(wn - ref_w) <= 12 * ULP * scale + 1e-30)
    np.testing.assert_allclose(m1, ref_m, rtol=4 * ULP)
    np.testing.assert_allclose(v1, ref_v, rtol=4 * ULP, atol=1e-44)
    np.testing.assert_allclose(ve1, ref_ve, rtol=8 * ULP, atol=1e-44)
    # both branches descend: the step opposes the gradient wherever g != 0
    step = wn.astype(np.float64) - W_HAND
    big = np.abs(step) > 1e-6 * np.abs(W_HAND)
    assert np.all(np.sign(step[big]) == -np.sign(G_HAND[big]))


def test_p4_ln2_enters_through_eps_scale():
    # with |g_e| comparable to eps the normalised exponent gradient keeps ln 2:
    # n = ln2 w g / (ln2 |w g| + eps); without ln 2 it would be 0.5 here.
    hp = oracle.hparams(lr_add=0.0, lr_mul=1e-3, eps=1e-8)
    w = np.array([1.0], F); g = np.array([1e-8], F); z = np.zeros(1, F)
    wn, *_ = oracle.update_elements(hp, 1, w, g, z, z, z)
    ge = math.log(2) * float(F(1e-8))
    n = ge / (ge + float(F(1e-8)))
    assert abs((float(wn[0]) - 1.0) - (-float(F(1e-3)) * n)) <= ULP   # binary32 resolution at 1
    assert abs(n - 0.5) > 0.05


def test_p4_second_step_closed_form():
    # the binary32 values the oracle receives
    b1, b2, eps = float(F(0.9)), float(F(0.999)), float(F(1e-8))
    lr_a, lr_m = float(F(1e-3)), float(F(1e-2))
    hp = oracle.hparams(lr_add=lr_a, lr_mul=lr_m)
    w0 = np.array([0.7, -0.05, 3.0, 1e-4], F)
    g1 = np.array([0.2, 1e-3, -0.4, 5e-3], F)
    g2 = np.array([-0.1, 2e-3, -0.3, -5e-3], F)
    z = np.zeros(4, F)
    w1, m1, v1, ve1 = oracle.update_elements(hp, 1, w0, g1, z, z, z)
    w2, m2, v2, ve2 = oracle.update_elements(hp, 2, w1, g2, m1, v1, ve1)
    W1 = w1.astype(np.float64); G1 = g1.astype(np.float64); G2 = g2.astype(np.float64)
    W0 = w0.astype(np.float64)
    # moments after two steps from zero
    M = b1 * (1 - b1) * G1 + (1 - b1) * G2
    V = b2 * (1 - b2) * G1 ** 2 + (1 - b2) * G2 ** 2
    GE1, GE2 = math.log(2) * W0 * G1, math.log(2) * W1 * G2
    VE = b2 * (1 - b2) * GE1 ** 2 + (1 - b2) * GE2 ** 2
    ua = -lr_a * (M / (1 - b1 ** 2)) / (np.sqrt(V / (1 - b2 ** 2)) + eps)
    n = GE2 / (np.sqrt(VE / (1 - b2 ** 2)) + eps)
    um = np.clip(-lr_m * n / np.maximum(np.abs(W1), 1e-8), -0.75, 0.75)
    ref = W1 + W1 * um + ua
    np.testing.assert_allclose(m2, M, rtol=8 * ULP)
    np.testing.assert_allclose(v2, V, rtol=8 * ULP)
    np.testing.assert_allclose(ve2, VE, rtol=16 * ULP)
    assert np.all(np.abs(w2 - ref) <= 16 * ULP * (np.abs(W1) + np.abs(ua) + np.abs(W1 * um)))


# ----------------------------------------------------------------------------
# P5: large-weight stall under BF16 storage
# ----------------------------------------------------------------------------
def _bf16_steps(w, g, hp, steps):
    wb = oracle.bf16_rne(np.array(w, F))
    gg = np.array(g, F)
    n = wb.size
    m = np.zeros(n, F); v = np.zeros(n, F); ve = np.zeros(n, F)
    for t in range(1, steps + 1):
        oracle.step_elements(hp, t, BF16, F32, F32, wb, gg, m, v, ve)
    return oracle.bf16_decode(wb)


def test_p5_additive_updates_vanish_at_large_weights_multiplicative_do_not():
    w, g = [256.0, -300.0], [0.5, -0.5]
    adam = _bf16_steps(w, g, oracle.hparams(lr_add=1e-3, lr_mul=0.0), 20)
    np.testing.assert_array_equal(adam, np.array([256.0, -300.0], F))   # stalled
    mp = _bf16_steps(w, g, oracle.hparams(lr_add=1e-3, lr_mul=2.0), 5)
    assert mp[0] < 256.0 and mp[1] > -300.0                               # moved


def test_p5_madam_cannot_escape_zero_madd_can():
    w, g = [0.0, 0.0], [1e-2, -1e-2]
    madam = _bf16_steps(w, g, oracle.hparams(lr_add=0.0, lr_mul=1e-2), 10)
    np.testing.assert_array_equal(madam, [0.0, 0.0])
    both = _bf16_steps(w, g, oracle.hparams(lr_add=1e-3, lr_mul=1e-2), 10)
    assert both[0] < 0 < both[1]


# ----------------------------------------------------------------------------
# P8: the log2 step cap as a clamp
# ----------------------------------------------------------------------------
@pytest.mark.parametrize("d", [1e-3, 0.05, 0.3, 0.8, 1.0, 3.0, math.inf])
def test_p8_step_cap_equals_clamp_of_um(d):
    s = oracle.scalars(oracle.hparams(dmult_max=d), 1)
    d = float(F(d))   # the binary32 cap the oracle receives
    hi_real = min(0.75, 2.0 ** d - 1.0)
    lo_real = max(-0.75, 2.0 ** -d - 1.0)
    # fp32 bounds are the innermost representable values
    assert float(s.hi) <= hi_real and float(np.nextafter(F(s.hi), F(1))) > hi_real
    assert float(s.lo) >= lo_real and float(np.nextafter(F(s.lo), F(-1))) < lo_real
    # literal path of Algorithm 2: clip to 0.75, log2, cap at d, exp2 - 1
    u = np.random.default_rng(3).uniform(-0.9, 0.9, 5000)
    lit = 2.0 ** np.clip(np.log2(1 + np.clip(u, -0.75, 0.75)), -d, d) - 1
    np.testing.assert_allclose(np.clip(u, lo_real, hi_real), lit, rtol=1e-12, atol=1e-15)


def test_p8_oracle_um_respects_cap():
    d = 0.1
    hp = oracle.hparams(lr_add=0.0, lr_mul=0.5, dmult_max=d)
    w = np.array([1.0, -1.0, 0.3, 2.0], F); g = np.array([1.0, 1.0, -1.0, 1e-3], F)
    z = np.zeros(4, F)
    wn, *_ = oracle.update_elements(hp, 1, w, g, z, z, z)
    de = np.log2(wn.astype(np.float64) / w)
    assert np.all(np.abs(de) <= d * (1 + 1e-5))
    assert np.all(np.abs(de) > 0.9 * d)   # capped, not just small


# ----------------------------------------------------------------------------
# P9 / P11: list split invariance and resume
# ----------------------------------------------------------------------------
def _tensors(sizes, seed, wdt=BF16):
    out = []
    for k, n in enumerate(sizes):
        w32 = _rand(n, seed + k, 0.02)
        w = oracle.bf16_rne(w32) if wdt == BF16 else oracle.e4m3_rne(w32 * 2.0 ** 11)
        out.append(dict(w=w, g=_rand(n, seed + 50 + k, 1e-3), m=np.zeros(n, F),
                        v=np.zeros(n, F), ve=np.zeros(n, F)))
    return out


def test_p9_split_at_multiple_of_8_is_bit_identical():
    hp = oracle.hparams(stochastic=1, seed=99)
    whole = _tensors([1000], 0)
    parts = [{k: a[:504].copy() for k, a in whole[0].items()},
             {k: a[504:].copy() for k, a in whole[0].items()}]
    for t in (1, 2, 3):
        oracle.step(whole, wdt=BF16, gdt=F32, mdt=F32, hp=hp, t=t)
        oracle.step(parts, wdt=BF16, gdt=F32, mdt=F32, hp=hp, t=t)
    for key in ("w", "m", "v", "ve"):
        np.testing.assert_array_equal(whole[0][key], np.concatenate([parts[0][key], parts[1][key]]))


@pytest.mark.parametrize("wdt", [BF16, E4M3])
def test_p11_resume_is_bit_exact(wdt):
    hp = oracle.hparams(stochastic=1, seed=5)
    a = _tensors([77, 1024, 5], 3, wdt)
    fa = oracle.fp8_init(a, [-11, -11, -11]) if wdt == E4M3 else None
    b = copy.deepcopy(a); fb = copy.deepcopy(fa)
    for t in range(1, 7):
        oracle.step(a, wdt=wdt, gdt=F32, mdt=F32, hp=hp, t=t, fp8_state=fa)
    for t in range(1, 4):
        oracle.step(b, wdt=wdt, gdt=F32, mdt=F32, hp=hp, t=t, fp8_state=fb)
    b = copy.deepcopy(b); fb = copy.deepcopy(fb)   # "checkpoint" and reload
    for t in range(4, 7):
        oracle.step(b, wdt=wdt, gdt=F32, mdt=F32, hp=hp, t=t, fp8_state=fb)
    for x, y in zip(a, b):
        for key in ("w", "m", "v", "ve"):
            np.testing.assert_array_equal(x[key], y[key])
    assert fa == fb


# ----------------------------------------------------------------------------
# P10: descent on a quadratic
# ----------------------------------------------------------------------------
def test_p10_descent_on_quadratic():
    n = 512
    rng = np.random.default_rng(4)
    target = rng.standard_normal(n).astype(F)
    w = (target + rng.standard_normal(n).astype(F) * F(2.0)).astype(F)
    hp = oracle.hparams(lr_add=1e-3, lr_mul=1e-3, beta1=0.0)
    m = np.zeros(n, F); v = np.zeros(n, F); ve = np.zeros(n, F)
    loss = [0.5 * float(np.sum((w.astype(np.float64) - target) ** 2))]
    for t in range(1, 31):
        g = (w - target).astype(F)
        oracle.step_elements(hp, t, F32, F32, F32, w, g, m, v, ve)
        loss.append(0.5 * float(np.sum((w.astype(np.float64) - target) ** 2)))
    assert all(b < a for a, b in zip(loss, loss[1:]))


# ----------------------------------------------------------------------------
# FP8 state bookkeeping
# ----------------------------------------------------------------------------
def test_fp8_state_tracks_amax_and_rescales():
    hp = oracle.hparams(lr_add=0.0, lr_mul=0.5)        # grow |w| fast
    ts = _tensors([256], 1, E4M3)
    ts[0]["g"][:] = -np.sign(oracle.e4m3_decode(ts[0]["w"])) * F(1e-2)
    st = oracle.fp8_init(ts, [-11])
    e_hist = [st[0][0]]
    for t in range(1, 8):
        before = st[0][1]
        oracle.step(ts, wdt=E4M3, gdt=F32, mdt=F32, hp=hp, t=t, fp8_state=st)
        e_hist.append(st[0][0])
        assert st[0][0] == oracle.fp8_next_exponent(before, e_hist[-2])
        dec = oracle.e4m3_decode(ts[0]["w"]).astype(np.float64) * 2.0 ** st[0][0]
        assert np.max(np.abs(dec)) <= 448.0 * 2.0 ** st[0][0]
    assert e_hist[-1] > e_hist[0]                        # the scale followed the growth
