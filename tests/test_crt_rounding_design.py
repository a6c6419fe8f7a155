"""The reconstruction's final rounding (one RNE rounding of X·2^E, §2.3
Phase 3) against the oracle's correctly rounded unscale.

The CUDA reconstruction holds X (|X| < 2^111) as a signed high word and a
low word.  For a normal result it takes the leading 64 bits with funnel
shifts, folds a sticky bit for the rest into bit 0 (below the rounding
position), lets the hardware u64 → f64 conversion round, and adds the
exponent to the bit pattern; subnormal, overflowing and small results take
a general rounding routine.  These CPU tests evaluate those steps with 32-
and 64-bit words (the hardware conversion is Python's correctly rounded
int → float) and compare each result bit for bit with the oracle.
"""
import math
import random
import struct

import pytest

from oracle import ozaki2 as orc

M32, M64 = (1 << 32) - 1, (1 << 64) - 1


def bits_of(x: float) -> int:
    return struct.unpack("<Q", struct.pack("<d", x))[0]


def from_bits(b: int) -> float:
    return struct.unpack("<d", struct.pack("<Q", b & M64))[0]


def clz32(w: int) -> int:
    return 32 - w.bit_length()


def round_to_double(x: int, sticky: bool, E: int, neg: bool) -> float:
    """Nearest double to ±(x + δ)·2^E, δ ∈ [0, 1) nonzero iff sticky."""
    sign = 1 << 63 if neg else 0
    if x == 0:
        return from_bits(sign)
    Lb = x.bit_length()
    top = Lb - 1 + E
    if top > 1023:
        return from_bits(sign | 0x7FF0000000000000)
    p = 53 if top >= -1022 else top + 1075
    sh = Lb - p
    if sh <= 0:
        q = (x << -sh) & M64
    elif p <= 0:
        below = (x & ((1 << (Lb - 1)) - 1)) != 0 or sticky
        q = 1 if (p == 0 and below) else 0
    else:
        q = x >> sh
        rbit = (x >> (sh - 1)) & 1
        st = sticky or (x & ((1 << (sh - 1)) - 1)) != 0
        if rbit and (st or (q & 1)):
            q += 1
    if q == 0:
        return from_bits(sign)
    if p < 53:
        return from_bits(sign | q)
    f = top
    if q >> 53:
        q >>= 1
        f += 1
    if f > 1023:
        return from_bits(sign | 0x7FF0000000000000)
    return from_bits(sign | ((f + 1023) << 52) | (q & ((1 << 52) - 1)))


def round_to_double_big(hi: int, lo: int, E: int, neg: bool) -> float:
    sh = hi.bit_length()
    top = ((hi << (64 - sh)) | (lo >> sh)) & M64
    return round_to_double(top, ((lo << (64 - sh)) & M64) != 0, E + sh, neg)


def finish_words(Hs: int, L: int, E: int) -> float:
    """Nearest double to X·2^E for X = Hs·2^64 + L (Hs signed, 0 ≤ L < 2^64)."""
    neg = Hs < 0
    hi, lo = Hs & M64, L
    if neg:
        lo = (-L) & M64
        hi = ((~hi) & M64) + (1 if L == 0 else 0)
    if hi == 0:
        return round_to_double(lo, False, E, neg)
    w3, w2, w1, w0 = hi >> 32, hi & M32, lo >> 32, lo & M32
    s = clz32(w3) if w3 else 32 + clz32(w2)
    e2 = E + 127 - s
    if e2 < -1022 or e2 > 1022:
        return round_to_double_big(hi, lo, E, neg)
    x3, x2, x1, x0 = (w2, w1, w0, 0) if s >= 32 else (w3, w2, w1, w0)
    sp = s & 31
    th = ((((x3 << 32) | x2) << sp) >> 32) & M32
    tl = ((((x2 << 32) | x1) << sp) >> 32) & M32
    sticky = (((x1 << sp) & M32) | x0) != 0
    top = (th << 32) | tl | (1 if sticky else 0)
    b = bits_of(float(top)) + ((E + 64 - s) << 52)   # the conversion rounds once
    return from_bits(b | ((1 << 63) if neg else 0))


def check(X: int, E: int):
    got = finish_words(X >> 64, X & M64, E)
    want = orc.unscale_one(X, E)
    assert bits_of(got) == bits_of(want) or (X == 0 and got == 0.0), (X, E, got, want)


def test_random_values_every_range():
    """|X| < 2^111 of every bit length, E from the overflow edge to far below
    the subnormal range."""
    rnd = random.Random(12)
    for _ in range(60_000):
        L = rnd.randint(1, 111)
        X = rnd.getrandbits(L) | (1 << (L - 1))
        X = -X if rnd.random() < 0.5 else X
        E = rnd.randint(-1250, 1030 - L)
        check(X, E)


def test_ties_and_sticky_bits():
    """Values exactly halfway between doubles (ties to even both ways), just
    above and below, with the tail bit far below the top word."""
    rnd = random.Random(13)
    for _ in range(20_000):
        L = rnd.randint(66, 111)
        q = rnd.getrandbits(53) | (1 << 52)
        half = 1 << (L - 54)
        base = q << (L - 53)
        for X in (base + half, base + half - 1, base + half + 1, base + 1, base):
            for sgn in (1, -1):
                check(sgn * X, rnd.randint(-1000, 1000 - L))


def test_subnormal_and_overflow_edges():
    for L in (1, 2, 53, 54, 64, 65, 100, 111):
        X = (1 << L) - 1
        for E in range(-1074 - L - 2, -1022 - L + 3):
            check(X, E)
            check(-X, E)
            check(1 << (L - 1), E)
        for E in range(1022 - L, 1026 - L):
            check(X, E)
            check(-X, E)
    check(0, 0)
    check(0, -2000)


def test_words_of_zero_low_part():
    """Negative X whose low word is zero (the two's complement carry)."""
    for L in range(65, 112, 7):
        for E in (-1100, -60, 0, 500):
            check(-(1 << L), E)
            check(-((1 << L) + (1 << 64)), E)
