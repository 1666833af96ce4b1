"""Pins of the oracle's NVFP4 storage: E2M1 payload (OCP FP4), one E4M3 scale
per 16 elements, one binary32 scale per tensor (Sec. 5.2's NVFP4 master
weights; the FP4 block-scale paragraph of the ablation appendix writes a
weight as payload times block scale)."""
from fractions import Fraction

import numpy as np
import pytest

import oracle
from oracle import F32

F = np.float32


def ocp_e2m1_value(code: int) -> Fraction:
    """OCP FP4 E2M1 from its bit fields: bias 1, exponent 0 is subnormal."""
    s, e, m = (code >> 3) & 1, (code >> 1) & 3, code & 1
    mag = Fraction(m, 2) if e == 0 else Fraction(2) ** (e - 1) * (1 + Fraction(m, 2))
    return -mag if s else mag


def test_e2m1_decode_is_the_ocp_definition():
    for c in range(16):
        assert Fraction(float(oracle.e2m1_decode(c)[0])) == ocp_e2m1_value(c)
    assert sorted({float(abs(ocp_e2m1_value(c))) for c in range(16)}) == [0, 0.5, 1, 1.5, 2, 3, 4, 6]


def _nearest_even(x: float) -> int:
    """Brute force over all 16 codes in exact rationals: the nearest value,
    ties to the code with mantissa bit 0; saturation at 6."""
    fx = Fraction(x)
    sign = 8 if np.signbit(x) else 0
    if abs(fx) >= 6:
        return sign | 7
    best = None
    for mag in range(8):
        d = abs(abs(fx) - abs(ocp_e2m1_value(mag)))
        key = (d, mag & 1)
        if best is None or key < best[0]:
            best = (key, mag)
    return sign | best[1]


def test_e2m1_rne_matches_brute_force_nearest_even():
    rng = np.random.default_rng(0)
    xs = np.concatenate([
        np.array([0.0, -0.0, 0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0, 6.0, 7.0, 1e9, -0.25, -5.0, -1e-30]),
        np.arange(0, 7, 1 / 64), (rng.random(3000) * 14 - 7),
    ]).astype(F)
    got = oracle.e2m1_rne(xs)
    want = np.array([_nearest_even(float(x)) for x in xs], np.uint8)
    np.testing.assert_array_equal(got, want)
    assert oracle.e2m1_rne([np.inf])[0] == 7 and oracle.e2m1_rne([-np.inf])[0] == 15
    assert oracle.e2m1_rne([np.nan])[0] == 0


def test_e2m1_sr_threshold_and_mean():
    """SR rounds away from zero iff r < floor(frac * 2^32): the mean over all
    r is within 2^-32 of a step of x, exact values never move."""
    rng = np.random.default_rng(1)
    for x in list(rng.random(300) * 12 - 6) + [0.5, 1.5, 3.0, -4.0, 0.0]:
        x = F(x)
        ax = Fraction(float(abs(x)))
        mags = [abs(ocp_e2m1_value(c)) for c in range(8)]
        lo = max(m for m in mags if m <= ax)
        hi = min([m for m in mags if m > ax], default=lo)
        if hi == lo:
            continue
        frac = (ax - lo) / (hi - lo)
        thr = int(frac * 2 ** 32)   # floor
        below = oracle.e2m1_sr([x, x], [max(thr - 1, 0), thr])
        if thr > 0:
            assert abs(ocp_e2m1_value(int(below[0]))) == hi
        assert abs(ocp_e2m1_value(int(below[1]))) == lo
        mean = lo + (hi - lo) * Fraction(thr, 2 ** 32)
        assert abs(mean - ax) <= (hi - lo) / 2 ** 32
    assert oracle.e2m1_sr([F(3.0)], [0xFFFFFFFF])[0] == 5       # exact values never move
    assert oracle.e2m1_sr([F(7.5)], [0])[0] == 7                 # saturation


def test_nvfp4_scale_code_defining_inequality_and_minimality():
    rng = np.random.default_rng(2)
    vals = oracle.e4m3_decode(np.arange(256, dtype=np.uint8))
    for _ in range(400):
        G = F(10.0 ** rng.uniform(-8, 0))
        amax = F(10.0 ** rng.uniform(-10, 2))
        c = oracle.nvfp4_scale_code(float(amax), float(G), 3)
        top = lambda k: F(6.0) * (F(vals[k]) * G)
        if top(126) >= amax:
            assert 1 <= c <= 126 and top(c) >= amax
            assert c == 1 or top(c - 1) < amax
        else:
            assert c == 126
    assert oracle.nvfp4_scale_code(0.0, 1e-3, 77) == 77


def _nvfp4_reference(hp, t, n, q0, bs0, G, g, gidx0):
    """The NVFP4 step composed from pinned pieces, block by block."""
    vals = oracle.e4m3_decode(np.arange(256, dtype=np.uint8))
    codes = oracle.nvfp4_unpack(q0, n)
    d_old = np.repeat((vals[bs0] * G).astype(F), 16)[:n]
    w = (oracle.e2m1_decode(codes) * d_old).astype(F)
    z = np.zeros(n, F)
    wn, m1, v1, ve1 = oracle.update_elements(hp, t, w, g, z, z, z)
    out, bs = np.zeros(n, np.uint8), bs0.copy()
    for b in range(bs0.size):
        sl = slice(16 * b, min(n, 16 * b + 16))
        fin = wn[sl][np.isfinite(wn[sl])]
        amax = float(np.max(np.abs(fin))) if fin.size else 0.0
        c = oracle.nvfp4_scale_code(amax, float(G), int(bs0[b]))
        bs[b] = c
        x = (wn[sl] / F(vals[c] * G)).astype(F)
        if hp.stochastic:
            r = oracle.rng_lanes(hp.seed, t, np.arange(gidx0 + sl.start, gidx0 + sl.stop, dtype=np.uint64),
                                 oracle.E4M3)
            out[sl] = oracle.e2m1_sr(x, r)
        else:
            out[sl] = oracle.e2m1_rne(x)
    return oracle.nvfp4_pack(out), bs, m1, v1, ve1


@pytest.mark.parametrize("stochastic", [0, 1])
@pytest.mark.parametrize("n", [1, 15, 16, 17, 33, 200, 1001])
def test_nvfp4_step_equals_composition_of_pinned_pieces(stochastic, n):
    rng = np.random.default_rng(n)
    G = F(0.02 / (6 * 448) * 4)
    w32 = (rng.standard_normal(n) * 0.02).astype(F)
    nb = -(-n // 16)
    bs0 = rng.integers(40, 110, nb).astype(np.uint8)
    vals = oracle.e4m3_decode(np.arange(256, dtype=np.uint8))
    d = np.repeat((vals[bs0] * G).astype(F), 16)[:n]
    q0 = oracle.nvfp4_pack(oracle.e2m1_rne(w32 / d))
    g = (rng.standard_normal(n) * 1e-3).astype(F)
    hp = oracle.hparams(stochastic=stochastic, seed=5, lr_mul=0.05)
    want = _nvfp4_reference(hp, 1, n, q0, bs0, G, g, gidx0=48)
    q, bs = q0.copy(), bs0.copy()
    m, v, ve = (np.zeros(n, F) for _ in range(3))
    oracle.step_nvfp4(hp, 1, F32, F32, n, q, bs, float(G), g.copy(), m, v, ve, gidx0=48)
    np.testing.assert_array_equal(oracle.nvfp4_unpack(q, n), oracle.nvfp4_unpack(want[0], n))
    np.testing.assert_array_equal(bs, want[1])
    for got, ref in zip((m, v, ve), want[2:]):
        np.testing.assert_array_equal(got.view(np.uint32), ref.view(np.uint32))


def test_nvfp4_blocks_fit_and_follow_growth():
    n = 256
    rng = np.random.default_rng(3)
    G = F(1e-4)   # block maxima near 0.05 sit mid-range (scale ~ 80 of 448)
    w32 = (rng.standard_normal(n) * 0.02).astype(F)
    bs = np.array([oracle.nvfp4_scale_code(float(np.abs(w32[i:i + 16]).max()), float(G), 1)
                   for i in range(0, n, 16)], np.uint8)
    vals = oracle.e4m3_decode(np.arange(256, dtype=np.uint8))
    q = oracle.nvfp4_pack(oracle.e2m1_rne(w32 / np.repeat((vals[bs] * G).astype(F), 16)))
    g = (-np.sign(w32) * 1e-2).astype(F)    # every weight grows
    m, v, ve = (np.zeros(n, F) for _ in range(3))
    hp = oracle.hparams(lr_add=0.0, lr_mul=0.3)
    b0 = bs.copy()
    for t in range(1, 6):
        oracle.step_nvfp4(hp, t, F32, F32, n, q, bs, float(G), g, m, v, ve)
        codes = oracle.nvfp4_unpack(q, n).reshape(-1, 16)
        assert np.all((codes & 7).max(axis=1) >= 4)       # each block uses the top of its range
    assert np.all(vals[bs] > vals[b0])


def test_nvfp4_dequant_is_payload_times_block_scale():
    rng = np.random.default_rng(4)
    n = 100
    codes = rng.integers(0, 16, n).astype(np.uint8)
    bs = rng.integers(1, 127, -(-n // 16)).astype(np.uint8)
    G = F(3.7e-4)
    got = oracle.dequant_nvfp4_bf16(n, oracle.nvfp4_pack(codes), bs, float(G))
    vals = oracle.e4m3_decode(np.arange(256, dtype=np.uint8))
    import torch
    import math
    # the sign bit gives -0 for code 8
    pay = np.array([math.copysign(float(abs(ocp_e2m1_value(int(c)))), -1.0 if c & 8 else 1.0) for c in codes], F)
    w = pay * np.repeat((vals[bs] * G).astype(F), 16)[:n]
    want = torch.from_numpy(w.astype(F)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(got, want)


def test_list_step_indexes_nvfp4_tensors_by_element_count():
    """Global indices follow element counts: an NVFP4 tensor of n elements
    (n/2 packed bytes) moves the next tensor's first index by n rounded up
    to a multiple of 8, so the next tensor draws the same random lanes as
    when stepped alone at that offset."""
    rng = np.random.default_rng(6)
    G = F(2.0 ** -12)
    mk = lambda n: dict(g=(rng.standard_normal(n) * 1e-3).astype(F), m=np.zeros(n, F), v=np.zeros(n, F),
                        ve=np.zeros(n, F))
    a = mk(37)
    a["bscale"] = np.full(3, 90, np.uint8)
    a["gscale"] = float(G)
    a["w"] = oracle.nvfp4_pack(rng.integers(0, 16, 37).astype(np.uint8))
    b = mk(50)
    b["w"] = oracle.bf16_rne((rng.standard_normal(50) * 0.02).astype(F))
    ref = {k: v.copy() if isinstance(v, np.ndarray) else v for k, v in b.items()}
    hp = oracle.hparams(stochastic=1, seed=9)
    oracle.step([a, b], wdt=[oracle.NVFP4, oracle.BF16], gdt=F32, mdt=F32, hp=hp, t=1)
    assert oracle.global_offsets([37, 50]) == [0, 40]
    oracle.step_elements(hp, 1, oracle.BF16, F32, F32, ref["w"], ref["g"], ref["m"], ref["v"], ref["ve"], gidx0=40)
    np.testing.assert_array_equal(b["w"], ref["w"])
