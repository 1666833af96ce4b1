"""Pins of the oracle's block-scaled E4M3 storage (FP16 power-of-two scales
per 32 elements; reading of Sec. 5.2 and the FP8-master figure) and of the
BF16 compute copy refreshed from the FP8 master each step."""
import numpy as np
import pytest
import torch

import oracle
from oracle import BF16, E4M3, E4M3_B32, F32

F = np.float32


def test_fp16_pow2_and_decode_match_torch():
    for k in range(-24, 16):
        want = torch.tensor(2.0 ** k, dtype=torch.float16).view(torch.int16).item() & 0xFFFF
        assert oracle.fp16_pow2(k) == want
    assert oracle.fp16_pow2(-30) == oracle.fp16_pow2(-24) and oracle.fp16_pow2(40) == oracle.fp16_pow2(15)
    h = np.arange(0, 1 << 16, 37, dtype=np.uint16)
    ref = torch.from_numpy(h.view(np.int16)).view(torch.float16).float().numpy()
    got = oracle.fp16_decode(h)
    ok = ~np.isnan(ref)
    np.testing.assert_array_equal(got[ok], ref[ok])
    assert np.all(np.isnan(got[~ok]))


def test_block_exponent_is_smallest_fitting_power_clamped():
    rng = np.random.default_rng(0)
    for a in (10.0 ** rng.uniform(-12, 8, 400)).astype(F):
        k = oracle.block_exponent(float(a), 3)
        if -24 < k < 15:
            assert float(a) <= 448 * 2.0 ** k and float(a) > 448 * 2.0 ** (k - 1)
    assert oracle.block_exponent(0.0, -7) == -7
    assert oracle.block_exponent(1e-30, 0) == -24 and oracle.block_exponent(1e30, 0) == 15


def test_dequant_bf16_matches_torch_casts():
    q = np.arange(256, dtype=np.uint8)
    dec = torch.from_numpy(q).view(torch.float8_e4m3fn).float()
    for e in (-11, -3, 0, 5):
        want = (dec * 2.0 ** e).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
        got = oracle.dequant_bf16(q, e)
        ok = ~torch.isnan(dec).numpy()
        np.testing.assert_array_equal(got[ok], want[ok])
    bs = np.array([oracle.fp16_pow2(k) for k in (-9, -2, 4, -20, 0, 1, -14, 15)], np.uint16)
    got = oracle.dequant_bf16(q, bscale=bs)
    scale = np.repeat(oracle.fp16_decode(bs), 32)
    want = (dec * torch.from_numpy(scale)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    ok = ~torch.isnan(dec).numpy()
    np.testing.assert_array_equal(got[ok], want[ok])


def _block_reference(hp, t, q0, bs0, g, gidx0):
    """The block step composed from pinned pieces: the per-element update,
    the exponent rule, the E4M3 encoders and the random lanes."""
    n = q0.size
    w = oracle.e4m3_decode(q0) * np.repeat(oracle.fp16_decode(bs0), 32)[:n]
    z = np.zeros(n, F)
    wn, m1, v1, ve1 = oracle.update_elements(hp, t, w, g, z, z, z)
    q, bs = np.zeros(n, np.uint8), bs0.copy()
    for b in range(bs0.size):
        sl = slice(32 * b, min(n, 32 * b + 32))
        fin = wn[sl][np.isfinite(wn[sl])]
        amax = float(np.max(np.abs(fin))) if fin.size else 0.0
        k_old = int(np.log2(oracle.fp16_decode(bs0[b:b + 1])[0]))
        k = oracle.block_exponent(amax, k_old)
        bs[b] = oracle.fp16_pow2(k)
        x = (wn[sl] * F(2.0 ** -k)).astype(F)
        if hp.stochastic:
            r = oracle.rng_lanes(hp.seed, t, np.arange(gidx0 + sl.start, gidx0 + sl.stop, dtype=np.uint64), E4M3)
            q[sl] = oracle.e4m3_sr(x, r)
        else:
            q[sl] = oracle.e4m3_rne(x)
    return q, bs, m1, v1, ve1


@pytest.mark.parametrize("stochastic", [0, 1])
@pytest.mark.parametrize("n", [1, 31, 32, 33, 200, 1000])
def test_block_step_equals_composition_of_pinned_pieces(stochastic, n):
    rng = np.random.default_rng(n)
    w32 = (rng.standard_normal(n) * 0.02 * 10.0 ** rng.uniform(-2, 2, n)).astype(F)
    bs0 = np.array([oracle.fp16_pow2(k) for k in rng.integers(-16, -6, -(-n // 32))], np.uint16)
    q0 = oracle.e4m3_rne(w32 / np.repeat(oracle.fp16_decode(bs0), 32)[:n])
    g = (rng.standard_normal(n) * 1e-3).astype(F)
    hp = oracle.hparams(stochastic=stochastic, seed=9, lr_mul=0.05)
    want = _block_reference(hp, 1, q0, bs0, g, gidx0=40)
    q, bs = q0.copy(), bs0.copy()
    m, v, ve = (np.zeros(n, F) for _ in range(3))
    oracle.step_block_e4m3(hp, 1, F32, F32, q, bs, g.copy(), m, v, ve, gidx0=40)
    np.testing.assert_array_equal(q, want[0])
    np.testing.assert_array_equal(bs, want[1])
    for got, ref in zip((m, v, ve), want[2:]):
        np.testing.assert_array_equal(got.view(np.uint32), ref.view(np.uint32))


def test_block_scales_follow_growth_and_fit_every_block():
    n = 256
    rng = np.random.default_rng(3)
    w32 = (rng.standard_normal(n) * 0.02).astype(F)
    bs = np.full(-(-n // 32), oracle.fp16_pow2(-12), np.uint16)
    q = oracle.e4m3_rne(w32 / F(2.0 ** -12))
    g = (-np.sign(w32) * 1e-2).astype(F)   # every weight grows
    m, v, ve = (np.zeros(n, F) for _ in range(3))
    hp = oracle.hparams(lr_add=0.0, lr_mul=0.5)
    k0 = np.log2(oracle.fp16_decode(bs))
    for t in range(1, 6):
        oracle.step_block_e4m3(hp, t, F32, F32, q, bs, g, m, v, ve)
        scale = np.repeat(oracle.fp16_decode(bs), 32)
        dec = oracle.e4m3_decode(q).astype(np.float64) * scale
        assert np.all(np.abs(dec) <= 448 * scale)
        assert np.all(np.abs(oracle.e4m3_decode(q)).reshape(-1, 32).max(1) > 224)  # scale is tight per block
    assert np.all(np.log2(oracle.fp16_decode(bs)) > k0)


def test_mixed_format_list_step():
    """A list with BF16 and block-scaled E4M3 tensors steps each by its own format,
    with global indices over the whole list."""
    rng = np.random.default_rng(5)
    sizes = [100, 64, 7, 96]
    fmts = [BF16, E4M3_B32, BF16, E4M3_B32]
    ts = []
    for n, f in zip(sizes, fmts):
        w32 = (rng.standard_normal(n) * 0.02).astype(F)
        d = dict(g=(rng.standard_normal(n) * 1e-3).astype(F), m=np.zeros(n, F), v=np.zeros(n, F), ve=np.zeros(n, F))
        if f == BF16:
            d["w"] = oracle.bf16_rne(w32)
        else:
            d["bscale"] = np.full(-(-n // 32), oracle.fp16_pow2(-11), np.uint16)
            d["w"] = oracle.e4m3_rne(w32 * F(2.0 ** 11))
        ts.append(d)
    ref = [{k: a.copy() for k, a in d.items()} for d in ts]
    hp = oracle.hparams(stochastic=1, seed=3)
    oracle.step(ts, wdt=fmts, gdt=F32, mdt=F32, hp=hp, t=1)
    offs = oracle.global_offsets(sizes)
    for k, (d, r) in enumerate(zip(ts, ref)):
        if fmts[k] == BF16:
            oracle.step_elements(hp, 1, BF16, F32, F32, r["w"], r["g"], r["m"], r["v"], r["ve"], gidx0=offs[k])
        else:
            oracle.step_block_e4m3(hp, 1, F32, F32, r["w"], r["bscale"], r["g"], r["m"], r["v"], r["ve"],
                                   gidx0=offs[k])
        for key in r:
            np.testing.assert_array_equal(d[key], r[key])
