"""Pins of the oracle's storage rounding (BF16 and E4M3) and FP8 scale rule.

- Round-to-nearest-even is pinned to torch's own casts (float32 -> bfloat16,
  float32 -> float8_e4m3fn), over strided sweeps of all binary32 patterns.
- E4M3 decoding is pinned to torch's float8_e4m3fn -> float32 on all 256 codes.
- Stochastic rounding is pinned to its definition by exact arithmetic: it never
  moves a representable value, it only ever returns one of the two neighbours,
  and the number of random words that round away from zero equals the exact
  fractional distance times 2^bits (exactly unbiased when enough bits are drawn).
- The scale rule is pinned by its defining inequality.
"""
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle


def _sweep(step, offset=0):
    """Every `step`-th binary32 bit pattern."""
    u = np.arange(offset, 1 << 32, step, dtype=np.uint64).astype(np.uint32)
    return u.view(np.float32)


# ----------------------------------------------------------------------------
# BF16
# ----------------------------------------------------------------------------
@pytest.mark.parametrize("offset", [0, 0x7FFF, 0x8000, 0x8001, 12345])
def test_bf16_rne_matches_torch(offset):
    x = _sweep(1 << 10, offset)
    x = x[~np.isnan(x)]
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = oracle.bf16_rne(x)
    np.testing.assert_array_equal(got, ref)


def test_bf16_nan_is_canonical():
    nans = np.array([0x7FC00000, 0xFFC00000, 0x7F800001, 0xFFFFFFFF, 0x7FFFFFFF],
                    np.uint32).view(np.float32)
    assert np.all(oracle.bf16_rne(nans) == 0x7FFF)
    assert np.all(oracle.bf16_sr(nans, np.full(5, 0xFFFF, np.uint32)) == 0x7FFF)


def test_bf16_sr_exact_on_representable():
    h = np.arange(0, 1 << 16, 7, dtype=np.uint32).astype(np.uint16)
    x = oracle.bf16_decode(h)
    keep = ~np.isnan(x)
    x, h = x[keep], h[keep]
    for r in (0, 1, 0x7FFF, 0xFFFF):
        np.testing.assert_array_equal(oracle.bf16_sr(x, np.full(x.size, r, np.uint32)), h)


def test_bf16_sr_is_exactly_unbiased():
    rng = np.random.default_rng(0)
    xs = rng.standard_normal(24) * 10.0 ** rng.integers(-30, 30, 24)
    xs = np.concatenate([xs, [3.4e38, -1.5e-40, 1e-45]]).astype(np.float32)
    r = np.arange(1 << 16, dtype=np.uint32)
    for x in xs:
        out = oracle.bf16_sr(np.full(r.size, x, np.float32), r)
        bits = int(np.float32(x).view(np.uint32))
        lo = bits >> 16
        assert set(np.unique(out).tolist()) <= {lo, lo + 1}
        n_away = int((out == lo + 1).sum())
        assert n_away == (bits & 0xFFFF)  # exact fractional distance x 2^16
        # expectation equals x exactly (rational arithmetic)
        f_lo = Fraction(float(np.uint32(lo << 16).view(np.float32)))
        if (lo + 1) & 0x7F80 != 0x7F80:
            f_hi = Fraction(float(np.uint32((lo + 1) << 16).view(np.float32)))
            mean = (f_lo * (65536 - n_away) + f_hi * n_away) / 65536
            assert mean == Fraction(float(x))


# ----------------------------------------------------------------------------
# E4M3
# ----------------------------------------------------------------------------
def test_e4m3_decode_matches_torch_all_codes():
    q = np.arange(256, dtype=np.uint8)
    ref = torch.from_numpy(q).view(torch.float8_e4m3fn).to(torch.float32).numpy()
    got = oracle.e4m3_decode(q)
    np.testing.assert_array_equal(np.isnan(got), np.isnan(ref))
    ok = ~np.isnan(ref)
    np.testing.assert_array_equal(got[ok].view(np.uint32), ref[ok].view(np.uint32))
    assert oracle.e4m3_decode(np.array([0x7E], np.uint8))[0] == 448.0
    assert oracle.e4m3_decode(np.array([0x01], np.uint8))[0] == 2.0 ** -9


@pytest.mark.parametrize("offset", [0, 0x7FFFF, 0x80000, 0x80001, 999])
def test_e4m3_rne_matches_torch_within_range(offset):
    x = _sweep(1 << 9, offset)
    x = x[np.isfinite(x) & (np.abs(x) <= 448.0)]
    ref = torch.from_numpy(x).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    got = oracle.e4m3_rne(x)
    np.testing.assert_array_equal(got, ref)


def test_e4m3_saturation_and_nan():
    x = np.array([448.0, 449.0, 464.0, 1e6, np.inf, -np.inf, -500.0, np.nan], np.float32)
    np.testing.assert_array_equal(oracle.e4m3_rne(x), [0x7E, 0x7E, 0x7E, 0x7E, 0x7E, 0xFE, 0xFE, 0x7F])
    r = np.full(x.size, 0, np.uint32)
    np.testing.assert_array_equal(oracle.e4m3_sr(x, r), [0x7E, 0x7E, 0x7E, 0x7E, 0x7E, 0xFE, 0xFE, 0x7F])


def test_e4m3_sr_exact_on_representable():
    q = np.arange(256, dtype=np.uint8)
    x = oracle.e4m3_decode(q)
    keep = ~np.isnan(x)
    for r in (0, 1, 0x80000000, 0xFFFFFFFF):
        np.testing.assert_array_equal(oracle.e4m3_sr(x[keep], np.full(keep.sum(), r, np.uint32)), q[keep])


def _neighbours(x):
    """E4M3 magnitudes just below/above |x| and the exact fraction, by search
    over the decoded code table (independent of the encoder's bit logic)."""
    mags = [Fraction(float(v)) for v in oracle.e4m3_decode(np.arange(0x7F, dtype=np.uint8))]
    ax = abs(Fraction(float(x)))
    lo_code = max(c for c, v in enumerate(mags) if v <= ax)
    hi = mags[lo_code + 1]
    return lo_code, (ax - mags[lo_code]) / (hi - mags[lo_code])


def test_e4m3_sr_threshold_is_floor_fraction_times_2p32():
    rng = np.random.default_rng(1)
    xs = np.concatenate([
        rng.uniform(-440, 440, 40), rng.uniform(-0.02, 0.02, 40),
        rng.uniform(-2.0 ** -6, 2.0 ** -6, 40), rng.uniform(-2.0 ** -9, 2.0 ** -9, 20),
        np.array([1e-30, -3e-41, 2.0 ** -10, 2.0 ** -10 + 2.0 ** -30])]).astype(np.float32)
    for x in xs:
        lo_code, frac = _neighbours(x)
        thr = int(frac * (1 << 32))  # floor
        sign = 0x80 if np.signbit(x) else 0

        def away(r):
            return int(oracle.e4m3_sr(np.array([x], np.float32), np.array([r], np.uint32))[0]) != (sign | lo_code)

        # decision is "r < thr": check both sides of the threshold and the ends
        if thr > 0:
            assert away(thr - 1) and away(0)
        assert not away(min(thr, 0xFFFFFFFF)) or thr > 0xFFFFFFFF
        assert not away(0xFFFFFFFF) or thr > 0xFFFFFFFF
        out0 = int(oracle.e4m3_sr(np.array([x], np.float32), np.array([0], np.uint32))[0])
        assert out0 in (sign | lo_code, sign | (lo_code + 1))


def test_e4m3_rne_ties_go_to_even():
    # midpoints between consecutive codes, at several binades
    q = np.arange(1, 0x7E, dtype=np.uint8)
    a = oracle.e4m3_decode(q).astype(np.float64)
    b = oracle.e4m3_decode(q + 1).astype(np.float64)
    mid = ((a + b) / 2).astype(np.float32)
    assert np.all(mid.astype(np.float64) == (a + b) / 2)
    got = oracle.e4m3_rne(mid)
    want = np.where(q % 2 == 0, q, q + 1).astype(np.uint8)
    np.testing.assert_array_equal(got, want)


# ----------------------------------------------------------------------------
# Scale rule (delayed per-tensor power-of-two scaling)
# ----------------------------------------------------------------------------
def test_fp8_next_exponent_is_smallest_fitting_power():
    rng = np.random.default_rng(2)
    amaxes = np.concatenate([10.0 ** rng.uniform(-20, 20, 300), [448.0, 449.0, 224.0, 1.0, 0.875]])
    for a in amaxes.astype(np.float32):
        k = oracle.fp8_next_exponent(float(a), 5)
        if -100 < k < 100:
            assert float(a) <= 448.0 * 2.0 ** k
            assert float(a) > 448.0 * 2.0 ** (k - 1)
    assert oracle.fp8_next_exponent(0.0, 17) == 17
    assert oracle.fp8_next_exponent(448.0, 3) == 0
    assert oracle.fp8_next_exponent(1e-38, 0) == -100
    assert oracle.fp8_next_exponent(3e38, 0) == 100
