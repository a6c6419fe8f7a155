"""Error budget of the reconstruction's two-word fast path (r ≤ 12).

The CUDA reconstruction finds X from 64-bit fixed-point sums: Y = Σ c_k F_k
mod 2^64 with F_k = round(2^64·y_k/m_k) approximates 2^64·X/M, the quotient
q = (S - X)/M comes from the 32-bit sum Σ c_k g_k with g_k =
round(2^18·y_k/m_k), and H = ⌊X/2^64⌋ is recovered from
Y·round(M/2^51)/2^115.  These CPU tests check,
with exact rational arithmetic on constants built here from their
definitions, that the worst case over all residues with |c_k| < m_k keeps
the error of that estimate well below the 1/2 that rounding H tolerates, and
that the quotient estimate keeps its margin too.  They also run the
word-level arithmetic on Python integers for random and extreme X.
"""
from fractions import Fraction
import random

import pytest

from oracle import ozaki2 as orc


def constants(r):
    mods = orc.moduli(r)
    M = 1
    for m in mods:
        M *= m
    out = []
    for m in mods:
        Mk = M // m
        y = pow(Mk % m, -1, m)
        F = ((y << 64) + m // 2) // m
        g = ((y << 18) + m // 2) // m
        out.append((m, y, Mk * y, F, g))
    return M, mods, out


@pytest.mark.parametrize("r", range(1, 13))
def test_fraction_error_budget(r):
    M, mods, cs = constants(r)
    assert M < 2 ** 112
    mh = (M + (1 << 50)) >> 51
    assert mh < 2 ** 61
    # |Y - 2^64·X/M| ≤ Σ |c_k|·|F_k - 2^64 y_k/m_k| with |c_k| ≤ m_k - 1.
    err_y = sum((m - 1) * abs(Fraction(F) - Fraction(y << 64, m)) for m, y, _, F, _ in cs)
    assert err_y <= Fraction(1, 2) * sum(m - 1 for m in mods)
    # H estimate in units of 2^64: Y error scaled by M/2^64, plus the rounding
    # of M/2^51 (|Y| < 2^63), the dropped low product and the floors of the
    # high product and of L/2^51 (one unit of 2^51 each).
    err_h = err_y * Fraction(M, 2 ** 64) / 2 ** 64 + Fraction(2 ** 63, 2 ** 64) * Fraction(1, 2) / 2 ** 13 \
        + Fraction(3, 2 ** 13)
    assert err_h < Fraction(1, 8), float(err_h)
    # Quotient estimate Σ c_k g_k/2^18 - Y/2^64 (q is an integer): error, with
    # the floors of g0/2^7 and Y/2^53, well below 1/2.
    err_q = sum((m - 1) * abs(Fraction(g) - Fraction(y << 18, m)) for m, y, _, _, g in cs) / 2 ** 18 \
        + (err_y + 1) / 2 ** 64 + Fraction(2, 2 ** 11)
    assert err_q < Fraction(1, 32), float(err_q)
    # The quotient sum is a 32-bit integer for any |c_k| < m_k.
    assert sum((m - 1) * g for m, _, _, _, g in cs) < 2 ** 31
    # The margin in Y (2^52) is far above its error.
    assert err_y < 2 ** 40


def word_path(c, r):
    """The fast path's word arithmetic on Python integers (two's complement
    words emulated with masks); returns X, or None where it defers."""
    M, mods, cs = constants(r)
    mask = (1 << 64) - 1
    Y = sum(ck * F for ck, (_, _, _, F, _) in zip(c, cs)) & mask
    Ys = Y - (1 << 64) if Y >> 63 else Y
    if abs(Ys if Ys >= 0 else ~Ys) >= (1 << 63) - (1 << 52):
        return None
    g0 = sum(ck * g for ck, (_, _, _, _, g) in zip(c, cs))
    assert -2 ** 31 <= g0 < 2 ** 31
    q = ((g0 >> 7) - (Ys >> 53) + 1024) >> 11
    L = (sum(ck * W for ck, (_, _, W, _, _) in zip(c, cs)) - q * M) & mask
    mh = (M + (1 << 50)) >> 51
    zh = (Ys * mh) >> 64
    H = (zh - (L >> 51) + 4096) >> 13
    return H * 2 ** 64 + L


@pytest.mark.parametrize("r", [1, 4, 8, 11, 12])
def test_word_path_recovers_x(r):
    M, mods, _ = constants(r)
    rng = random.Random(r)
    lo, hi = -(M // 2), M - M // 2 - 1
    xs = [0, 1, -1, lo, hi, lo + (M >> 12) + 1, hi - (M >> 12) - 1]
    xs += [rng.randrange(lo, hi + 1) for _ in range(300)]
    xs += [rng.randrange(max(lo, -(1 << 64)), min(hi, 1 << 64) + 1) for _ in range(100)]
    deferred = 0
    for x in xs:
        c = [int(orc.centred(x % m, m)) for m in mods]
        # also a non-centred representative with |c| < m
        c2 = [ck + m if ck < 0 else ck - m if ck > 0 else ck for ck, m in zip(c, mods)]
        for cc in (c, c2):
            got = word_path(cc, r)
            if got is None:
                deferred += 1
                assert abs(x) > M // 2 - (M >> 11)
            else:
                assert got == x, (r, x)
    assert deferred <= 8


def w128_constants(r):
    """W_k = (M/m_k)·y_k, F_k = round(2^32·y_k/m_k) and coff_k = m_k·⌈2^15/m_k⌉,
    built here from their definitions."""
    mods = orc.moduli(r)
    M = 1
    for m in mods:
        M *= m
    out = []
    for m in mods:
        Mk = M // m
        y = pow(Mk % m, -1, m)
        out.append((m, Mk * y, ((y << 32) + m // 2) // m, m * -(-32768 // m)))
    return M, mods, out


def w128_path(c, r):
    """The r = 13 fast path's word arithmetic on Python integers: word sums
    of u_k = c_k + coff_k over W_k's 32-bit words, the 32.32 quotient sum,
    and S - q·M mod 2^128 read as a signed word.  Returns X, or None where
    the quotient is ambiguous."""
    M, mods, cs = w128_constants(r)
    m64, m32 = (1 << 64) - 1, (1 << 32) - 1
    a = [0, 0, 0]
    a3 = 0
    Q = 1 << 31
    for ck, (m, W, F, coff) in zip(c, cs):
        u = ck + coff
        assert 0 <= u < 2 ** 16.1
        for j in range(3):
            a[j] += u * ((W >> (32 * j)) & m32)
        a3 = (a3 + u * ((W >> 96) & m32)) & m32
        Q += u * F
    assert max(a) < 2 ** 52 and Q < 2 ** 64
    frac = Q & m32
    if frac < (1 << 19) or frac > m32 - (1 << 19):
        return None
    q = Q >> 32
    assert q < 2 ** 20
    lo = (a[0] + (a[1] << 32)) & m64
    hi = ((a[1] >> 32) + a[2] + (a3 << 32) + (1 if lo < a[0] else 0)) & m64
    pl = (q * (M & m64)) & m64
    ph = (q * ((M >> 64) & m64) + ((q * (M & m64)) >> 64)) & m64
    L = (lo - pl) & m64
    H = (hi - ph - (1 if lo < pl else 0)) & m64
    X = (H << 64) | L
    return X - (1 << 128) if X >> 127 else X


def test_w128_range():
    """r = 13 is the one count past the two-word path whose X fits a signed
    128-bit word with room: 2^112 < M < 2^121; r = 14 does not fit."""
    M13, _, cs = w128_constants(13)
    assert 2 ** 112 < M13 < 2 ** 121
    assert all(W < 2 ** 128 for _, W, _, _ in cs)
    assert w128_constants(14)[0] > 2 ** 128


def test_w128_path_recovers_x():
    r = 13
    M, mods, _ = w128_constants(r)
    rng = random.Random(13)
    lo, hi = -(M // 2), M - M // 2 - 1
    xs = [0, 1, -1, lo, hi, lo + 1, hi - 1, (1 << 64), -(1 << 64), (1 << 64) - 1, -(1 << 119), (1 << 119)]
    xs += [rng.randrange(lo, hi + 1) for _ in range(400)]
    xs += [rng.randrange(-(1 << 70), 1 << 70) for _ in range(100)]
    xs += [lo + rng.randrange(M >> 12) for _ in range(50)] + [hi - rng.randrange(M >> 12) for _ in range(50)]
    deferred = 0
    for x in xs:
        c = [int(orc.centred(x % m, m)) for m in mods]
        # also other int16 representatives of the same residues
        c2 = [ck + m if ck < 0 else ck - m if ck > 0 else ck for ck, m in zip(c, mods)]
        c3 = [ck + m * ((32767 - ck) // m) if ck < -100 else ck - m * ((ck + 32768) // m)
              for ck, m in zip(c, mods)]  # representatives at the ends of the int16 range
        for cc in (c, c2, c3):
            assert all(-2 ** 15 <= v < 2 ** 15 for v in cc)
            got = w128_path(cc, r)
            if got is None:
                deferred += 1
                assert abs(x) > M // 2 - (M >> 12), x
            else:
                assert got == x, x
    assert deferred <= 3 * 106  # only the 100 band samples and the ends of the range


def w160_path(c, r):
    """The r = 14..16 fast path's word arithmetic on Python integers: word
    sums of u_k over W_k's words 0..3 and word 4 mod 2^32, the 32.32 quotient
    sum, S' - q·M mod 2^160 read as a signed word.  Returns X, or None where
    the quotient is ambiguous."""
    M, mods, cs = w128_constants(r)
    m64, m32 = (1 << 64) - 1, (1 << 32) - 1
    a = [0, 0, 0, 0]
    a4 = 0
    Q = 1 << 31
    for ck, (m, W, F, coff) in zip(c, cs):
        u = ck + coff
        for j in range(4):
            a[j] += u * ((W >> (32 * j)) & m32)
        a4 = (a4 + u * ((W >> 128) & m32)) & m32
        Q += u * F
    assert max(a) < 2 ** 53 and Q < 2 ** 64
    frac = Q & m32
    if frac < (1 << 19) or frac > m32 - (1 << 19):
        return None
    q = Q >> 32
    assert q < 2 ** 21
    lo = (a[0] + (a[1] << 32)) & m64
    s1 = (a[1] >> 32) + a[2] + (1 if lo < a[0] else 0)
    assert s1 < 2 ** 64
    mid = (s1 + (a[3] << 32)) & m64
    top = ((a[3] >> 32) + a4 + (1 if mid < s1 else 0)) & m32
    P = q * M
    X = ((top << 128) | (mid << 64) | lo) - P
    X &= (1 << 160) - 1
    return X - (1 << 160) if X >> 159 else X


def test_w160_range():
    """r = 14..16 fit a signed 160-bit word: M < 2^148, W_k < 2^160, and the
    top word of M (bits 128 and up) is below 2^20."""
    for r in (14, 15, 16):
        M, _, cs = w128_constants(r)
        assert 2 ** 121 < M < 2 ** 148
        assert all(W < 2 ** 160 for _, W, _, _ in cs)
        assert (M >> 128) < 2 ** 20


@pytest.mark.parametrize("r", [14, 16])
def test_w160_path_recovers_x(r):
    M, mods, _ = w128_constants(r)
    rng = random.Random(r)
    lo, hi = -(M // 2), M - M // 2 - 1
    xs = [0, 1, -1, lo, hi, lo + 1, hi - 1, 1 << 64, -(1 << 64), 1 << 128, -(1 << 128), (1 << 128) - 1]
    xs += [rng.randrange(lo, hi + 1) for _ in range(300)]
    xs += [rng.randrange(-(1 << 100), 1 << 100) for _ in range(60)]
    xs += [lo + rng.randrange(M >> 12) for _ in range(30)] + [hi - rng.randrange(M >> 12) for _ in range(30)]
    for x in xs:
        c = [int(orc.centred(x % m, m)) for m in mods]
        c2 = [ck + m if ck < 0 else ck - m if ck > 0 else ck for ck, m in zip(c, mods)]
        c3 = [ck + m * ((32767 - ck) // m) if ck < -100 else ck - m * ((ck + 32768) // m)
              for ck, m in zip(c, mods)]
        for cc in (c, c2, c3):
            got = w160_path(cc, r)
            if got is None:
                assert abs(x) > M // 2 - (M >> 12), x
            else:
                assert got == x, x
