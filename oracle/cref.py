"""Independent high-accuracy references for AB (TEST INFRASTRUCTURE ONLY).

These define no result of the method; they measure its error, the quantity
named by §2.6 "Error Analysis" (u plus the quantisation of Eq. scale).

* :func:`exact_entry` -- the exact rational Σ_l A_il B_lj, by scaling every
  double to an integer mantissa times a power of two and summing Python ints.
* :func:`dot2` -- Ogita, Rump and Oishi's compensated dot product ("Accurate
  sum and dot product", SIAM J. Sci. Comput. 26(6), 2005), kept as an
  unevaluated pair (hi, lo) so that the error |C - (hi + lo)| can be formed
  without a final rounding of the reference.  TwoProduct uses Dekker's split
  (Veltkamp constant 2^27 + 1); TwoSum is Knuth's.
"""
from __future__ import annotations

import math
from fractions import Fraction

import numpy as np


def exact_entry(a_row, b_col) -> Fraction:
    """Σ_l a_l b_l exactly (finite inputs)."""
    total = 0
    emin = None
    terms = []
    for a, b in zip(a_row, b_col):
        a = float(a)
        b = float(b)
        if a == 0.0 or b == 0.0:
            continue
        ma, ea = math.frexp(a)
        mb, eb = math.frexp(b)
        ia = int(ma * 2**53)
        ib = int(mb * 2**53)
        e = ea + eb - 106
        terms.append((ia * ib, e))
        emin = e if emin is None else min(emin, e)
    if not terms:
        return Fraction(0)
    for v, e in terms:
        total += v << (e - emin)
    return Fraction(total) * Fraction(2) ** emin


def _two_sum(a, b):
    s = a + b
    bb = s - a
    err = (a - (s - bb)) + (b - bb)
    return s, err


_SPLIT = 134217729.0  # 2^27 + 1


def _split(a):
    c = _SPLIT * a
    hi = c - (c - a)
    return hi, a - hi


def _two_product(a, b):
    p = a * b
    ah, al = _split(a)
    bh, bl = _split(b)
    err = al * bl - (((p - ah * bh) - al * bh) - ah * bl)
    return p, err


def dot2(A, B, rows=None):
    """(hi, lo) with hi + lo ≈ AB[rows, :] to about (k u)^2 |A||B| + u^2|AB|.

    Vectorised over output entries; loops over k.  Inputs must be finite and
    small enough that the split does not overflow (|x| < 2^995).
    """
    A = np.asarray(A, dtype=np.float64)
    B = np.asarray(B, dtype=np.float64)
    if rows is not None:
        A = A[rows]
    m, k = A.shape
    n = B.shape[1]
    s = np.zeros((m, n))
    c = np.zeros((m, n))
    with np.errstate(over="ignore", invalid="ignore"):
        for l in range(k):
            p, pe = _two_product(A[:, l:l + 1], B[l:l + 1, :])
            s, se = _two_sum(s, p)
            c = c + (pe + se)
    return s, c


def abs_product(A, B, rows=None):
    """|A||B| (rounded; used only as the error normaliser)."""
    A = np.asarray(A, dtype=np.float64)
    if rows is not None:
        A = A[rows]
    return np.abs(A) @ np.abs(np.asarray(B, dtype=np.float64))


def scaled_error(C, A, B, rows=None):
    """max_ij |C - AB|_ij / (|A||B|)_ij over the given rows (0/0 counts as 0)."""
    hi, lo = dot2(A, B, rows)
    Cs = np.asarray(C)[rows] if rows is not None else np.asarray(C)
    err = np.abs((Cs - hi) - lo)
    nrm = abs_product(A, B, rows)
    with np.errstate(invalid="ignore", divide="ignore"):
        q = np.where(nrm > 0, err / nrm, np.where(err > 0, np.inf, 0.0))
    return float(q.max(initial=0.0))
