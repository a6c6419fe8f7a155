"""The deconstruction's 32-bit integer arithmetic against the oracle.

The deconstruction (Algorithm 1, quantise and deconstruct; §2.5) computes
each entry's centred residues with 32-bit integer steps:

* a branch-free truncating quantisation: the significand shifted up by 10
  and back down with clamping funnel shifts, the sign applied as a two's
  complement, for scales d ≤ 1083 (and d = -4096 for rows that are zero);
* Ã split into 21-bit limbs, Ã = v0 + v1·2^21 + v2·2^42 with v2 signed,
  the lowest biased by 2^31, summed per modulus with the centred limb
  weights 2^21 mod m and 2^42 mod m, so the sum lies in (0, 2^32);
* a multiply-high quotient by ⌈2^32/m⌉ that may be one too large, so the
  remainder lies in [-m, m) and indexes a table of 2m entries rotated by
  the bias (nonsquare moduli);
* for square moduli, an added constant that makes the remainder the centred
  residue plus ⌊m/2⌋, then balanced base-s digits by a multiply-high.

These CPU tests evaluate those steps with 32-bit wrap-around, with every
constant recomputed from its definition, and compare them with the oracle's
quantiser, centred residues and digit functions.
"""
import numpy as np
import pytest

from oracle import ozaki2 as orc

M32 = np.uint64(0xFFFFFFFF)
BIAS = 1 << 31          # the limb-sum bias
LIMB = 21               # limb width
TZ_FAST_MAX_D = 1083    # largest scale the branch-free path takes


def u64(x):
    return np.asarray(x, dtype=np.uint64)


def funnel_right_clamped(lo, hi, sh):
    """Low word of (hi:lo) >> min(sh, 32)."""
    s = np.minimum(sh, np.uint64(32))
    return ((hi << np.uint64(32)) | lo) >> s & M32


def split_word(tl, th):
    """The kernel's limbs (w0, w1, w2) of the two's complement word th:tl
    (tl unsigned 32-bit, th signed)."""
    mask = np.uint64((1 << LIMB) - 1)
    w0 = (tl & mask) | np.uint64(BIAS)
    w1 = ((u64(th & 0xFFFFFFFF) << np.uint64(32) | tl) >> np.uint64(LIMB)) & mask
    w2 = np.asarray(th, dtype=np.int64) >> (2 * LIMB - 32)
    return w0, w1, w2


def quantise_tz_limbs(x, d):
    """The kernel's limbs of trunc(x·2^d)."""
    bits = np.asarray(x, dtype=np.float64).view(np.uint64)
    hi, lo = bits >> np.uint64(32), bits & M32
    E = ((hi >> np.uint64(20)) & np.uint64(0x7FF)).astype(np.int64)
    mh = (hi & np.uint64(0xFFFFF)) | np.where(E != 0, np.uint64(0x100000), np.uint64(0))
    r = u64((10 + 1075 - np.maximum(E, 1) - np.asarray(d, dtype=np.int64)) & 0xFFFFFFFF)
    ph = ((mh << np.uint64(10)) | (lo >> np.uint64(22))) & M32
    pl = (lo << np.uint64(10)) & M32
    wide = r >= np.uint64(32)
    x1 = np.where(wide, np.uint64(0), ph)
    x0 = np.where(wide, ph, pl)
    rr = np.where(wide, r - np.uint64(32), r)
    al = funnel_right_clamped(x0, x1, rr)
    ah = funnel_right_clamped(x1, np.uint64(0), rr)
    neg = (hi >> np.uint64(31)) != 0
    sgn = np.where(neg, M32, np.uint64(0))
    t = (((ah ^ sgn) << np.uint64(32)) | (al ^ sgn)) + neg.astype(np.uint64)  # two's complement negation
    tl = t & M32
    th = (t >> np.uint64(32)).astype(np.int64)
    th = np.where(th >= 1 << 31, th - (1 << 32), th)
    return split_word(tl, th)


def limbs_of(At):
    """The same limbs taken straight from Ã (|Ã| < 2^62)."""
    At = np.asarray(At, dtype=np.int64)
    return split_word(u64(At & 0xFFFFFFFF), At >> 32)


def value_of(w0, w1, w2):
    return (w0.astype(np.int64) - BIAS) + (w1.astype(np.int64) << LIMB) + (w2 << (2 * LIMB))


def centred_weight(j, m):
    return int(orc.centred(pow(2, LIMB * j, m), m))


def limb_sum(w0, w1, w2, m, extra=0):
    """Y = w0 + extra + w1·c1 + w2·c2 with the centred weights c_j = 2^21j
    mod m, wrapped to 32 bits, and the same sum without wrapping."""
    c1, c2 = centred_weight(1, m), centred_weight(2, m)
    exact = w0.astype(np.int64) + extra + w1.astype(np.int64) * c1 + w2 * c2
    Y = (w0 + np.uint64(extra) + w1 * np.uint64(c1 & 0xFFFFFFFF) + u64(w2 & 0xFFFFFFFF) * np.uint64(c2 & 0xFFFFFFFF)) & M32
    return Y, exact


def mulhi(a, b):
    return (u64(a) * u64(b)) >> np.uint64(32)


def residue_samples(rng, n=200_000):
    lim = (1 << 62) - 1
    At = rng.integers(-lim, lim, size=n, dtype=np.int64)
    small = rng.integers(-(1 << 20), 1 << 20, size=n // 4, dtype=np.int64)
    edges = np.array([0, 1, -1, lim, -lim, 1 << 32, -(1 << 32), (1 << 48) - 1, -(1 << 48),
                      (1 << 16) - 1, -(1 << 16)], dtype=np.int64)
    return np.concatenate([At, small, edges])


def test_tz_quantiser_limbs():
    """Normal, subnormal and zero entries at scales that keep |Ã| < 2^62, at
    d = 1083 and at the zeroing scale -4096."""
    rng = np.random.default_rng(5)
    n = 200_000
    sig = rng.uniform(0.5, 1.0, size=n) * rng.choice([-1.0, 1.0], size=n)
    e = rng.integers(-1074, 1024, size=n)
    x = np.ldexp(sig, e)
    x = np.concatenate([x, np.ldexp(rng.uniform(-1, 1, size=n // 10), -1074 + rng.integers(0, 52, size=n // 10)),
                        np.array([0.0, -0.0, 5e-324, -5e-324, np.finfo(float).max, -np.finfo(float).tiny])])
    ex = np.frexp(x)[1]                       # |x| < 2^ex
    dmax = np.minimum(TZ_FAST_MAX_D, 62 - ex)  # trunc(|x|·2^d) < 2^62
    d = np.maximum(dmax - rng.integers(0, 120, size=x.size), -1100)
    d = np.where(rng.random(x.size) < 0.02, -4096, d)
    d = np.where(x == 0, rng.integers(-1100, TZ_FAST_MAX_D + 1, size=x.size), d)
    got = value_of(*quantise_tz_limbs(x, d))
    want = orc.quantise(x[:, None], d)[:, 0]
    assert np.array_equal(got, want)


def test_limb_split_round_trip():
    rng = np.random.default_rng(6)
    At = residue_samples(rng)
    assert np.array_equal(value_of(*limbs_of(At)), At)


@pytest.mark.parametrize("m", [m for m in orc.moduli(16) if not orc.square_base(m)])
def test_nonsquare_table_index(m):
    """Y - qm lies in [-m, m), and entry m + (Y - qm) of the rotated table
    (entry i: the residue (i - 2^31) mod m) is Ã mod m."""
    rng = np.random.default_rng(m)
    At = residue_samples(rng)
    Y, exact = limb_sum(*limbs_of(At), m)
    assert np.all((exact > 0) & (exact < 1 << 32))
    assert np.array_equal(Y.astype(np.int64), exact)
    magic = -(-(1 << 32) // m)
    assert magic < 1 << 32
    q = mulhi(Y, magic).astype(np.int64)
    off = exact - q * m
    assert np.all((off >= -m) & (off < m))
    entry = m + off
    assert np.array_equal(np.mod(entry - BIAS, m), np.mod(At, m))


@pytest.mark.parametrize("m", [m for m in orc.moduli(16) if not orc.square_base(m)] + [1089, 529])
def test_limb_sum_stays_in_range_at_the_extremes(m):
    """The sum's bounds at the limbs' extreme values: v0 ∈ [0, 2^21),
    v1 ∈ [0, 2^21), v2 ∈ [-2^20, 2^20), with the square moduli's added
    constant below m."""
    c1, c2 = centred_weight(1, m), centred_weight(2, m)
    lo = BIAS + min(0, c1) * ((1 << LIMB) - 1) + min(-c2 * (1 << 20), c2 * ((1 << 20) - 1))
    hi = BIAS + (1 << LIMB) - 1 + m + max(0, c1) * ((1 << LIMB) - 1) + max(-c2 * (1 << 20), c2 * ((1 << 20) - 1))
    assert 0 < lo and hi < 1 << 32


def square_digits_fp(u, s, h0, h1):
    """The kernel's FP32 digits of u = c + h0 + s·h1 for s ≠ 32: with the
    float ub = 1.5·2^23 + u and cs = ⌈2^17/s⌉/2^17, one fused multiply-add
    rounded down, t = RD(ub·cs + (1.5·2^23 - 96·⌈2^17/s⌉)), which is
    1.5·2^23 + ⌊u·⌈2^17/s⌉/2^17⌋ (the grid at 1.5·2^23 is the integers);
    d1 = t - (1.5·2^23 + h1), d0 = (u - h0 - s·h1) - s·d1."""
    c17 = -(-(1 << 17) // s)
    base = 3 << 22
    addend = base - 96 * c17
    assert 0 < addend < 1 << 24 and 96 * c17 * (1 << 17) == base * c17   # 1.5·2^23·cs = 96·c17
    ub = base + np.asarray(u, dtype=object)
    t = np.array([(int(x) * c17 + addend * (1 << 17)) // (1 << 17) for x in ub], dtype=np.int64)  # RD of the exact value
    d1 = t - (base + h1)
    d0 = (u - h0 - s * h1) - s * d1
    return d0, d1, t


@pytest.mark.parametrize("m", [m for m in orc.moduli(16) if orc.square_base(m)])
def test_square_digits(m):
    """The kernel's square digits from the limbs of Ã equal the oracle's
    digits of the centred residue: the sum with the added constant, the
    corrected remainder, then a shift and mask for s = 32 and the FP32
    form for the other bases."""
    s = orc.square_base(m)
    H = m // 2
    E = (H - BIAS) % m
    h0 = s // 2
    h1 = -(-(H - h0) // s)
    shift = h0 + s * h1 - H
    assert shift >= 0
    rng = np.random.default_rng(m)
    At = residue_samples(rng)
    Y, exact = limb_sum(*limbs_of(At), m, extra=E)
    assert np.all((exact > 0) & (exact < 1 << 32))
    assert np.array_equal(Y.astype(np.int64), exact)
    q = mulhi(Y, -(-(1 << 32) // m)).astype(np.int64)
    off = exact - q * m
    assert np.all((off >= -m) & (off < m))
    off = np.where(off < 0, off + m, off)
    u = off + shift
    if s == 32:
        d0, d1 = (u & 31) - h0, (u >> 5) - h1
    else:
        d0, d1, _ = square_digits_fp(u, s, h0, h1)
    w0, w1 = orc.square_digits(orc.centred(At, m), s)
    assert np.array_equal(d0, w0) and np.array_equal(d1, w1)


@pytest.mark.parametrize("m", [m for m in orc.moduli(16) if orc.square_base(m) and orc.square_base(m) != 32])
def test_square_digits_by_fp32_fma(m):
    """The FP32 form of the square digits over every centred residue: the
    rounded-down fused multiply-add gives ⌊u/s⌋ exactly, the digits match
    the oracle's, and every operand and result is an integer below 2^24."""
    s = orc.square_base(m)
    H = m // 2
    h0 = s // 2
    h1 = -(-(H - h0) // s)
    cs = np.arange(-H, m - H)
    u = cs + h0 + s * h1
    base = 3 << 22
    assert u.min() >= 0 and (base + u).max() < 1 << 24
    d0, d1, t = square_digits_fp(u, s, h0, h1)
    assert np.array_equal(t - base, u // s)
    w0, w1 = orc.square_digits(cs, s)
    assert np.array_equal(d0, w0) and np.array_equal(d1, w1)
    assert np.abs(d0).max() <= 16 and np.abs(d1).max() <= 16
