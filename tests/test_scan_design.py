"""The scan key and the magnitude-plane code (Algorithm 1 "scan the exponent
spans"; §2.4 "+1" pass) against the oracle, from the bits of each double.

The scan kernels reduce each row to the maximum of a per-entry key: 0 for a
zero, the frexp exponent plus 2048 for a finite nonzero entry (the bit
length of the significand for a subnormal), and 2^20 for Inf or NaN.  The
magnitude pass writes the E4M3 code of 2^max(-c, ⌈log2|x|⌉ - e), reading
⌈log2|x|⌉ of a normal double off its exponent field and whether its fraction
is zero.  These CPU tests evaluate both from the bit patterns as the kernels
do and compare them with the oracle's exponents and E4M3 encoder.
"""
import numpy as np
import pytest

from oracle import ozaki2 as orc


def scan_key(x: float) -> int:
    b = int(np.float64(x).view(np.uint64))
    E = (b >> 52) & 0x7FF
    mant = b & ((1 << 52) - 1)
    if E == 0x7FF:
        return 1 << 20
    if E == 0:
        return 0 if mant == 0 else mant.bit_length() - 1074 + 2048
    return E - 1022 + 2048


def e4m3_pow2(q: int) -> int:
    return (q + 7) << 3 if q >= -6 else 1 << (q + 9)


def magnitude_code(x: float, ex: int, c: int) -> int:
    b = int(np.float64(x).view(np.uint64))
    E = (b >> 52) & 0x7FF
    frac = (b & ((1 << 52) - 1)) != 0
    if E == 0x7FF:
        return 0
    if E == 0:
        if not frac:
            return 0
        return e4m3_pow2(max(-c, int(orc.ceil_log2_abs(x)) - ex))
    return e4m3_pow2(max(-c, E - 1023 + (1 if frac else 0) - ex))


def sample_doubles(rng, n):
    sig = rng.uniform(0.5, 1.0, size=n) * rng.choice([-1.0, 1.0], size=n)
    x = np.ldexp(sig, rng.integers(-1074, 1025, size=n))
    powers = np.ldexp(1.0, rng.integers(-1074, 1024, size=n // 10))
    sub = np.ldexp(rng.uniform(-1, 1, size=n // 10), -1022 - rng.integers(0, 53, size=n // 10))
    special = np.array([0.0, -0.0, np.inf, -np.inf, np.nan, 5e-324, np.finfo(float).max,
                        np.finfo(float).tiny, -np.finfo(float).tiny / 2])
    return np.concatenate([x, powers, -powers, sub, special])


def test_scan_key():
    x = sample_doubles(np.random.default_rng(21), 50_000)
    got = np.array([scan_key(v) for v in x])
    finite_nz = np.isfinite(x) & (x != 0)
    want = np.where(~np.isfinite(x), 1 << 20, np.where(finite_nz, orc.frexp_exponent(np.where(finite_nz, x, 1.0)) + 2048, 0))
    assert np.array_equal(got, want)
    # the row maximum of the keys is the row exponent of the oracle's scan
    rows = x[: 49_000].reshape(-1, 7)
    rows = rows[np.isfinite(rows).all(axis=1)]
    e, _, nz = orc.scan_rows(rows)
    kmax = np.array([max(scan_key(v) for v in r) for r in rows])
    assert np.array_equal(np.where(nz, kmax - 2048, 0), np.where(nz, e, 0))


@pytest.mark.parametrize("c", [0, 3, 6, 9])
def test_magnitude_code(c):
    rng = np.random.default_rng(22 + c)
    x = sample_doubles(rng, 20_000)
    x = x[np.isfinite(x)]
    ex = orc.frexp_exponent(np.abs(x)) + rng.integers(0, 12, size=x.size)   # a row exponent ≥ the entry's
    got = np.array([magnitude_code(v, int(e), c) for v, e in zip(x, ex)])
    q = orc.magnitude_exponents(x[:, None], ex, c)[:, 0]
    want = np.array([0 if qi == -10**6 else orc.e4m3_encode_power_of_two(int(qi)) for qi in q])
    assert np.array_equal(got, want)
