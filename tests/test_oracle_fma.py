"""Pin of reading R3: where the canonical binary32 sequence takes a product
and a sum together, it rounds once (a fused multiply-add), not twice.

The paper writes the update of Algorithm 1 in real arithmetic and fixes
only that the step is computed in binary32 and the result rounded into
storage (Sec. 5.1, App. B).  The sequence the oracle and the kernel follow
fuses five sites:

    mu'   = fma(b1, mu, (1-b1) g)
    nu'   = fma(b2, nu, (1-b2) g^2)
    nu_e' = fma(b2, nu_e, (1-b2) g_e^2)
    den   = fma(sqrt(nu'), c2, eps)        (and the same for nu_e')
    w'    = fma(w, u_m, w) + u_a

Each test below evaluates the fused operation exactly, in rational
arithmetic rounded once to binary32 (round to nearest, ties to even), and
the rest of the sequence with numpy binary32 operations, which are
correctly rounded.  It asserts that the oracle returns that value, and that
on the same inputs a twice-rounded version of the site gives a different
result for many elements: an "unfused" edit of any one site fails here.
"""
from fractions import Fraction

import numpy as np
import pytest

import oracle

F = np.float32


def round_f32(x: Fraction) -> np.float32:
    """An exact rational rounded once to binary32, nearest with ties to
    even (subnormals, overflow to infinity)."""
    if x == 0:
        return F(0.0)
    sign = -1 if x < 0 else 1
    a = abs(x)
    e = a.numerator.bit_length() - a.denominator.bit_length()  # 2^e <= a < 2^(e+2)
    if a < Fraction(2) ** e:
        e -= 1
    if a >= Fraction(2) ** (e + 1):
        e += 1
    q = Fraction(2) ** (max(e, -126) - 23)  # spacing of binary32 numbers at a
    n = a / q
    k = n.numerator // n.denominator
    rem = n - k
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and k % 2 == 1):
        k += 1
    r = k * q
    if r >= Fraction(2) ** 128:
        return F(sign * np.inf)
    return F(sign * float(r))


def fma(a, b, c) -> np.float32:
    return round_f32(Fraction(float(a)) * Fraction(float(b)) + Fraction(float(c)))


def unfused(a, b, c) -> np.float32:
    return F(F(F(a) * F(b)) + F(c))


def model(s, w, g, m, v, ve, site_unfused=None):
    """The canonical per-element sequence in binary32, with the named site
    rounded twice instead of once (None: all fused)."""
    def f(site, a, b, c):
        return unfused(a, b, c) if site == site_unfused else fma(a, b, c)
    m1 = f("m", s.b1, m, F(F(s.omb1) * g))
    v1 = f("v", s.b2, v, F(F(s.omb2) * F(g * g)))
    den_a = f("den_a", np.sqrt(v1), s.c2, s.eps)
    ua = F(F(F(s.ka) * m1) / den_a)
    ge = F(F(F(s.ln2) * w) * g)
    ve1 = f("ve", s.b2, ve, F(F(s.omb2) * F(ge * ge)))
    den_e = f("den_e", np.sqrt(ve1), s.c2, s.eps)
    n = F(ge / den_e)
    um = F(F(F(s.km) * n) / max(abs(w), F(s.tau)))
    um = F(max(F(s.lo), min(um, F(s.hi))))
    wn = F(f("w", w, um, w) + ua)
    return wn, m1, v1, ve1


def _inputs(n, seed):
    r = np.random.default_rng(seed)
    w = (r.standard_normal(n) * 0.02).astype(F)
    g = (r.standard_normal(n) * 1e-3).astype(F)
    m = (r.standard_normal(n) * 1e-3).astype(F)
    v = (np.abs(r.standard_normal(n)) * 1e-6).astype(F)
    ve = (np.abs(r.standard_normal(n)) * 1e-12).astype(F)
    return w, g, m, v, ve


# Which output shows each site: the moments directly; the denominators and
# the combine through the binary32 weight, with inputs that let a one-ulp
# change reach it:
# - den_a: w = 0, so g_e = 0, u_m = -0 and w' = 0 + u_a = u_a exactly;
# - den_e and the combine: eta_a = 0 (u_a = -0) and eta_m = 0.01, so that
#   |u_m| is of order 0.5 and w u_m moves w' at its own last bits.
SITES = [
    ("m", 1, {}, False),
    ("v", 2, {}, False),
    ("ve", 3, {}, False),
    ("den_a", 0, {}, True),
    ("den_e", 0, dict(lr_add=0.0, lr_mul=0.01), False),
    ("w", 0, dict(lr_add=0.0, lr_mul=0.01), False),
]


@pytest.mark.parametrize("site,out,hp_kw,zero_w", SITES, ids=[x[0] for x in SITES])
def test_oracle_rounds_each_fused_site_once(site, out, hp_kw, zero_w):
    n = 400
    w, g, m, v, ve = _inputs(n, seed=[x[0] for x in SITES].index(site) + 1)
    if zero_w:
        w[:] = 0.0
    hp = oracle.hparams(**hp_kw)
    t = 3
    s = oracle.scalars(hp, t)
    got = oracle.update_elements(hp, t, w, g, m, v, ve)[out]
    differ = 0
    for i in range(n):
        fused_val = model(s, w[i], g[i], m[i], v[i], ve[i])[out]
        twice_val = model(s, w[i], g[i], m[i], v[i], ve[i], site_unfused=site)[out]
        assert got[i].view(np.uint32) == fused_val.view(np.uint32), (site, i, got[i], fused_val)
        differ += int(twice_val.view(np.uint32) != fused_val.view(np.uint32))
    # the inputs do tell the two readings apart
    assert differ >= 10, (site, differ)


def test_round_f32_agrees_with_numpy_on_exact_binary64_values():
    """The test's own rounding: float64 values (exact rationals) rounded to
    binary32 by numpy's correctly rounded conversion, including ties and
    subnormals."""
    r = np.random.default_rng(5)
    xs = list(r.standard_normal(2000) * 10.0 ** r.integers(-44, 38, 2000))
    # ties (halfway between binary32 neighbours: to even), subnormal ties, the largest finite
    xs += [1.0 + 2.0 ** -24, 1.0 + 3 * 2.0 ** -24, -(1.0 + 2.0 ** -24), 2.0 ** -149 * 0.5, 2.0 ** -149 * 1.5,
           3.4028234663852886e38]
    for x in xs:
        assert round_f32(Fraction(float(x))).view(np.uint32) == F(x).view(np.uint32), x
