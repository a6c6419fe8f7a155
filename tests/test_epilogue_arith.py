"""The residue GEMM's FP32 reduction arithmetic against the integer definition.

The epilogue (and the split-K fold) reduce integer-valued FP32 sums mod m
with the 1.5·2^23 rounding constant and fused multiply-adds.  These CPU tests
evaluate the same steps, in the same order and precision, with each fused
multiply-add computed exactly in extended precision and rounded once to
FP32, and compare them with the centred residue of the oracle (reading
R-centre):

* loose_mod(x) for integers |x| ≤ 2^24: congruent to x and below 1.5m;
* centred_small(v) for every integer |v| < 2^16: the centred residue;
* the full recombination of two accumulators |a0|, |a1| ≤ 2^24 (Eq.
  sq-shortcut for squares, the merged form 16·acc0 - 15·acc1 for nonsquare
  moduli), and the two short-slab forms for combined sums below 2^24.

The samples for |x| ≤ 2^24 hold every integer within one of a rounding
boundary (q·m and q·m ± m/2 for every q in range), the extremes, and a
strided sweep.
"""
import numpy as np
import pytest

from oracle import ozaki2 as orc

if np.finfo(np.longdouble).nmant < 63:
    pytest.skip("needs an extended long double to evaluate FP32 fused multiply-adds exactly",
                allow_module_level=True)

F32, LD = np.float32, np.longdouble
MAGIC = F32(12582912.0)  # 1.5·2^23


def fmaf(a, b, c):
    """FP32 fused multiply-add: the exact a·b + c (the products here have at
    most 48 significant bits and the sums span at most 58), rounded once."""
    a, b, c = (np.asarray(t, dtype=F32).astype(LD) for t in (a, b, c))
    return (a * b + c).astype(F32)


def consts(m):
    mf = F32(m)
    return mf, F32(1.0) / mf, F32(m - 1 - m // 2)


def loose_mod(x, mf, inv):
    q = fmaf(x, inv, MAGIC) - MAGIC
    return fmaf(-q, mf, x)


def centred_small(v, mf, inv, hi):
    q = fmaf(v, inv, MAGIC) - MAGIC
    r = fmaf(-q, mf, v)
    return np.where(r > hi, r - mf, r)


def combine(a0, a1, square, s, mf, inv, hi):
    r0, r1 = loose_mod(a0, mf, inv), loose_mod(a1, mf, inv)
    v = fmaf(F32(s), r1, r0) if square else fmaf(F32(16), r0, F32(-15) * r1)
    return centred_small(v, mf, inv, hi)


def combine_short(a0, a1, square, s, mf, inv, hi):
    v = fmaf(F32(s), a1, a0) if square else fmaf(F32(16), a0, F32(-15) * a1)
    return centred_small(loose_mod(v, mf, inv), mf, inv, hi)


def combine_short1(a0, a1, square, s, mf, inv, hi):
    v = fmaf(F32(s), a1, a0) if square else fmaf(F32(16), a0, F32(-15) * a1)
    r = loose_mod(v, mf, inv)
    r = np.where(r > hi, r - mf, r)
    return np.where(r < hi + F32(1) - mf, r + mf, r)


def boundary_samples(m, limit=2 ** 24):
    """Integers |x| ≤ limit near every rounding boundary of x/m, plus the
    extremes and a strided sweep."""
    q = np.arange(-(limit // m) - 1, limit // m + 2, dtype=np.int64)
    h = m // 2
    offs = np.array([-h - 1, -h, -h + 1, -1, 0, 1, m - 1 - h - 1, m - 1 - h, m - h], dtype=np.int64)
    x = (q[:, None] * m + offs[None, :]).ravel()
    edge = np.arange(0, 1024, dtype=np.int64)
    x = np.concatenate([x, limit - edge, -limit + edge, np.arange(-limit, limit + 1, 9973, dtype=np.int64)])
    return x[np.abs(x) <= limit]


@pytest.mark.parametrize("m", orc.moduli(16))
def test_loose_mod(m):
    mf, inv, _ = consts(m)
    x = boundary_samples(m)
    r = loose_mod(x.astype(F32), mf, inv).astype(np.int64)
    assert np.all((x - r) % m == 0)
    assert np.all(2 * np.abs(r) < 3 * m)


@pytest.mark.parametrize("m", orc.moduli(16))
def test_centred_small_exhaustive(m):
    mf, inv, hi = consts(m)
    v = np.arange(-(2 ** 16) + 1, 2 ** 16, dtype=np.int64)
    got = centred_small(v.astype(F32), mf, inv, hi).astype(np.int64)
    assert np.array_equal(got, orc.centred(v, m))


@pytest.mark.parametrize("m", orc.moduli(16))
def test_accumulator_recombination(m):
    """Random and extreme accumulator pairs, |a0|, |a1| ≤ 2^24."""
    mf, inv, hi = consts(m)
    s = orc.square_base(m)
    rng = np.random.default_rng(m)
    a0 = rng.integers(-(2 ** 24), 2 ** 24 + 1, size=200_000)
    a1 = rng.integers(-(2 ** 24), 2 ** 24 + 1, size=200_000)
    ext = np.array([-(2 ** 24), -(2 ** 24) + 1, -1, 0, 1, 2 ** 24 - 1, 2 ** 24], dtype=np.int64)
    a0 = np.concatenate([a0, np.repeat(ext, ext.size)])
    a1 = np.concatenate([a1, np.tile(ext, ext.size)])
    got = combine(a0.astype(F32), a1.astype(F32), s is not None, s or 16, mf, inv, hi).astype(np.int64)
    want = orc.centred(a0 + s * a1 if s else 16 * a0 - 15 * a1, m)
    assert np.array_equal(got, want)


@pytest.mark.parametrize("m", orc.moduli(16))
def test_short_slab_forms(m):
    """Combined sums v below 2^24 (the short-slab bound): accumulator pairs
    whose v is every boundary sample, and random pairs inside the bound."""
    mf, inv, hi = consts(m)
    s = orc.square_base(m)
    x = boundary_samples(m, 2 ** 24 - 1)
    rng = np.random.default_rng(1000 + m)
    if s:  # v = a0 + s·a1
        b1, b0 = np.floor_divide(x, s), np.mod(x, s)
        a1 = rng.integers(-(2 ** 24) // (2 * s), 2 ** 24 // (2 * s), size=100_000)
        a0 = rng.integers(-(2 ** 23) + 1, 2 ** 23, size=100_000)
    else:  # v = 16·a0 - 15·a1
        b1 = np.mod(x, 16)
        b0 = np.floor_divide(x, 16) + b1
        a1 = rng.integers(-(2 ** 23) // 15, 2 ** 23 // 15, size=100_000)
        a0 = rng.integers(-(2 ** 23) // 16, 2 ** 23 // 16, size=100_000)
    a0 = np.concatenate([b0, a0])
    a1 = np.concatenate([b1, a1])
    v = a0 + s * a1 if s else 16 * a0 - 15 * a1
    assert np.all(np.abs(v) < 2 ** 24) and np.array_equal(v[:x.size], x)
    want = orc.centred(v, m)
    for form in (combine_short, combine_short1):
        got = form(a0.astype(F32), a1.astype(F32), s is not None, s or 16, mf, inv, hi).astype(np.int64)
        assert np.array_equal(got, want), form.__name__
