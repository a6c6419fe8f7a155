"""Exactness budget of the residue GEMM's FP32 accumulators and epilogue.

The tensor cores accumulate integer plane products in FP32, which is exact
while every partial sum stays below 2^24 (Eq. accum-exact).  These CPU tests
derive the digit extremes from the oracle's own digit functions (§2.5) and
check the inequalities the CUDA epilogue relies on:

* K-slabs: 32768 k-steps for square moduli (two accumulators), 4096 for the
  merged nonsquare ones (the paper's maximum merged term 4095);
* the short-slab path, which combines the accumulators before reducing them:
  |acc0 + s·acc1| < 2^24 for K ≤ 896 (square) and |16·acc0 - 15·acc1| < 2^24
  for K ≤ 128 (nonsquare).
"""
import numpy as np
import pytest

from oracle import ozaki2 as orc

K_SLAB_SQUARE, K_SLAB_MERGED = 32768, 4096
SHORT_SQUARE, SHORT_NONSQUARE = 7 * 128, 1 * 128


def digits(m):
    d = orc.centred(np.arange(m), m)
    s = int(round(m ** 0.5))
    if s * s == m:
        d0, d1 = orc.square_digits(d, s)
        return "square", s, d0, d1
    d0, d1 = orc.nonsquare_digits(d)[:2]
    return "nonsquare", 16, d0, d1


@pytest.mark.parametrize("m", orc.moduli(16))
def test_accumulator_terms(m):
    kind, s, d0, d1 = digits(m)
    if kind == "square":
        t0 = np.abs(np.outer(d0, d0)).max()                       # acc0 term d0·e0
        t1 = np.abs(np.outer(d1, d0) + np.outer(d0, d1)).max()    # acc1 term d1·e0 + d0·e1
        assert t0 <= 256 and t1 <= 512
        assert K_SLAB_SQUARE * max(t0, t1) <= 2 ** 24
        assert SHORT_SQUARE * (t0 + s * t1) < 2 ** 24
    else:
        sig = np.abs(np.outer(d0 + d1, d0 + d1)).max()          # acc0 term (d0+d1)(e0+e1)
        mer = np.abs(np.outer(d0, d0) - 16 * np.outer(d1, d1)).max()   # merged acc1 term
        assert sig <= 484 and mer <= 4095
        assert K_SLAB_MERGED * max(sig, mer) <= 2 ** 24
        assert SHORT_NONSQUARE * (16 * sig + 15 * mer) < 2 ** 24


def test_merged_term_extreme_is_the_papers():
    worst = max(np.abs(np.outer(d0, d0) - 16 * np.outer(d1, d1)).max()
                for kind, _, d0, d1 in map(digits, orc.moduli(16)) if kind == "nonsquare")
    assert worst == 4095
