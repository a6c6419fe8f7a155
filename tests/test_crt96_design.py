"""The fused kernel's 96-bit CRT estimate (r = 11, 12), on the CPU.

The fused residue-GEMM + reconstruction kernel folds each modulus's residue
into one fixed-point sum per output and estimates X from it: with
F_k = round(2^96·y_k/m_k), Y = Σ c_k F_k mod 2^96 (a signed word) is
2^96·X/M + D with |D| ≤ Σ|c_k|/2, and P = ⌊|Y|·M/2^96⌋ (partial products of
32-bit words below 2^64 dropped) is within a host-computed bound err of |X|.
The rounding of X·2^E is taken from P when no midpoint between doubles lies
within err of P; otherwise an exact path runs.  These tests build the
constants here from their definitions, check the bound against the worst
residues, emulate the word arithmetic on Python integers, and compare every
value the fast path returns with the correctly rounded X·2^E (float of an
exact rational), including X placed next to midpoints.  The kernel sees
centred residues; the cases with other representatives check the same
arithmetic under the wider bound those need.
"""
from fractions import Fraction
import math
import random

import pytest

from oracle import ozaki2 as orc

MASK32 = (1 << 32) - 1


def signed_low(v):
    lo = v & MASK32
    return lo - (1 << 32) if lo >> 31 else lo


def constants(r):
    mods = orc.moduli(r)
    M = 1
    for m in mods:
        M *= m
    ks = []
    for m in mods:
        y = pow((M // m) % m, -1, m)
        F = ((y << 96) + m // 2) // m
        f0 = signed_low(F)
        F1 = (F - f0) >> 32
        f1 = signed_low(F1)
        f2 = ((F1 - f1) >> 32) & MASK32
        assert f0 + (f1 << 32) + (f2 << 64) == F
        ks.append((m, y, F, f0, f1, f2))
    return M, mods, ks


def err_bound(M, mods, centred):
    cmax = sum(m // 2 for m in mods) if centred else 32768 * len(mods)
    return -(-(cmax * ((M >> 64) + 1)) // (1 << 33)) + 6


def s32(v):
    v &= MASK32
    return v - (1 << 32) if v >> 31 else v


def fast_path(c, E, r, err):
    """The CUDA fast path on Python integers; the double, or None (defer)."""
    M, mods, ks = constants(r)
    a0 = sum(ck * f0 for ck, (_, _, _, f0, _, _) in zip(c, ks))
    a1 = sum(ck * f1 for ck, (_, _, _, _, f1, _) in zip(c, ks))
    a2 = sum(ck * f2 for ck, (_, _, _, _, _, f2) in zip(c, ks)) & MASK32
    assert -2 ** 63 <= a0 < 2 ** 63 and -2 ** 63 <= a1 < 2 ** 63
    s1 = (a0 >> 32) + a1
    w0, w1 = a0 & MASK32, s1 & MASK32
    w2 = ((s1 >> 32) + a2) & MASK32
    Y = (w2 << 64) | (w1 << 32) | w0
    neg = Y >> 95
    mag = ((1 << 96) - Y) % (1 << 96) if neg else Y
    y0, y1, y2 = mag & MASK32, (mag >> 32) & MASK32, mag >> 64
    if y2 >= 0x7FFFFFFF:
        return None
    m0, m1, m2, m3 = [(M >> (32 * i)) & MASK32 for i in range(4)]
    assert M >> 128 == 0 and m3 < 2 ** 16
    c2 = ((y0 * m2) >> 32) + ((y1 * m1) >> 32) + ((y2 * m0) >> 32)
    P = y0 * m3 + c2 + y1 * m2 + y2 * m1 + ((y1 * m3 + y2 * m2) << 32) + ((y2 * m3) << 64)
    assert P >> 128 == 0
    ph = P >> 64
    lz = 64 - ph.bit_length()
    if lz > 43:
        return None
    sh = 64 - lz
    u = sh - 21
    ew = (err >> u) + 2
    W = (P >> u) & MASK32
    if ew >= 1 << 29 or ((W - 0x80000000 + ew) & MASK32) <= 2 * ew:
        return None
    top = (P >> sh) | (W >> 31)
    assert top >> 63 == 1
    e2 = 127 - lz + E
    if e2 < -1022 or e2 > 1022:
        return None
    v = math.ldexp(float(top), E + sh)
    return -v if neg else v


def exact(x, E):
    return float(Fraction(x) * Fraction(2) ** E)


def residues(x, mods, centred=True):
    c = [int(orc.centred(x % m, m)) for m in mods]
    if not centred:   # other representatives: shift each by a multiple of m inside int16
        c = [ck + m * ((31 * (k + 1) + x) % (32768 // m) - (16384 // m)) for k, (ck, m) in enumerate(zip(c, mods))]
        assert all(-32768 <= ck < 32768 for ck in c)
    return c


@pytest.mark.parametrize("r", [11, 12])
def test_bound_holds_for_the_worst_residues(r):
    """|D|·M/2^96 + the dropped products stays inside err for residues at
    their largest magnitude with the signs of the rounding errors of F_k."""
    M, mods, ks = constants(r)
    for centred in (True, False):
        cmax = [m // 2 if centred else 32768 for m in mods]
        D = sum(cm * abs(Fraction(F) - Fraction(y << 96, m)) for cm, (m, y, F, _, _, _) in zip(cmax, ks))
        assert D * Fraction(M, 2 ** 96) + 5 <= err_bound(M, mods, centred)
    if r == 12:
        assert err_bound(M, mods, True) < 2 ** 28


@pytest.mark.parametrize("r", [11, 12])
def test_fast_path_rounds_like_the_exact_value(r):
    M, mods, _ = constants(r)
    rng = random.Random(1000 + r)
    lo, hi = -(M // 2), M - M // 2 - 1
    taken = 0
    cases = []
    for _ in range(1500):
        bits = rng.randrange(max(1, M.bit_length() - 30), M.bit_length())
        x = rng.randrange(1 << (bits - 1), 1 << bits) * rng.choice((1, -1))
        cases.append(max(lo, min(hi, x)))
    cases += [rng.randrange(lo, hi + 1) for _ in range(100)] + [0, 1, -1, lo, hi, 2 ** 60 + 1, -(2 ** 70)]
    for x in cases:
        for centred in (True, False):
            E = rng.randrange(-1200, 1000) - x.bit_length() // 2
            got = fast_path(residues(x, mods, centred), E, r, err_bound(M, mods, centred))
            if got is None:
                continue
            taken += 1
            assert got == exact(x, E) and math.copysign(1, got) == math.copysign(1, exact(x, E) or 1.0)
    assert taken > 1500


def test_midpoints_defer_and_everything_else_is_exact():
    """X placed at and around midpoints between doubles: the fast path either
    defers or gives the correctly rounded value."""
    r = 12
    M, mods, _ = constants(r)
    err = err_bound(M, mods, True)
    rng = random.Random(7)
    deferred = 0
    for b in (86, 88, 90, 96, 100, 105, 109, 110):
        q = b - 53
        for _ in range(40):
            base = rng.randrange(1 << 52, 1 << 53) << q
            for off in (0, 1, -1, err // 2, -err // 2, err, -err, 3 * err, -3 * err, 1 << (q - 3)):
                x = (base + (1 << (q - 1)) + off) * rng.choice((1, -1))
                if abs(x) >= M // 2:
                    continue
                E = -(b + 20)
                got = fast_path(residues(x, mods), E, r, err)
                if got is None:
                    deferred += 1
                    continue
                assert got == exact(x, E), (b, off)
    assert deferred > 0


@pytest.mark.parametrize("r", [11, 12])
def test_typical_outputs_take_the_fast_path(r):
    """Outputs whose |X| is within 2^28 of the scale bound M/4 (the dense
    problems' typical range) almost never defer."""
    M, mods, _ = constants(r)
    err = err_bound(M, mods, True)
    rng = random.Random(11 + r)
    top = M.bit_length() - 2
    xs = [rng.randrange(1 << (top - 28), 1 << top) * rng.choice((1, -1)) for _ in range(2000)]
    deferred = sum(fast_path(residues(x, mods), -top - 10, r, err) is None for x in xs)
    assert deferred <= 1


def test_small_and_subnormal_results_defer():
    r = 12
    M, mods, _ = constants(r)
    err = err_bound(M, mods, True)
    for x in (0, 5, -(2 ** 40), 2 ** 80):
        assert fast_path(residues(x, mods), -10, r, err) is None
    x = 2 ** 100 + 12345
    assert fast_path(residues(x, mods), -1200, r, err) is None      # subnormal result
    assert fast_path(residues(x, mods), 1000, r, err) is None       # overflow
    assert fast_path(residues(x, mods), -50, r, err) == exact(x, -50)


def test_tie_in_the_leading_word_rounds_up():
    """P above the midpoint by less than one unit of its leading 64-bit word:
    that word alone is an exact tie, and the path must still round up."""
    x, E, r = 4583600681551543933728663411072, -577, 11
    M, mods, _ = constants(r)
    got = fast_path(residues(x, mods), E, r, err_bound(M, mods, True))
    assert got == exact(x, E)
    rng = random.Random(5)
    for _ in range(300):
        q = rng.randrange(40, 57)
        x = (rng.randrange(1 << 52, 1 << 53) << q) + (1 << (q - 1)) + rng.randrange(1 << 30, 1 << (q - 2))
        if x >= M // 2:
            continue
        got = fast_path(residues(x, mods), -100, r, err_bound(M, mods, True))
        assert got is None or got == exact(x, -100)


def test_planted_mistake_is_caught():
    """A bound 2^12 times too small lets a near-midpoint X through wrongly:
    the comparison with the exact rounding must notice."""
    r = 12
    M, mods, _ = constants(r)
    err = err_bound(M, mods, True)
    rng = random.Random(3)
    wrong = 0
    for _ in range(3000):
        q = 100 - 53
        x = (rng.randrange(1 << 52, 1 << 53) << q) + (1 << (q - 1)) + rng.randrange(-err, err)
        got = fast_path(residues(x, mods), -120, r, err >> 12)
        if got is not None and got != exact(x, -120):
            wrong += 1
    assert wrong > 0
