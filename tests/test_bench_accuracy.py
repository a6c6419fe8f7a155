"""The bench's error measurement (sampled entries of C - AB summed exactly)
against exact rational arithmetic: a measurement the bench reports, so it is
pinned here on the CPU."""
from fractions import Fraction

import numpy as np

import bench
import workloads as wl
from oracle import cref


def exact_scaled_error(C, A, B, rows, cols):
    worst = 0.0
    for i in rows:
        for j in cols:
            err = abs(Fraction(float(C[i, j])) - cref.exact_entry(A[i], B[:, j]))
            nrm = float(np.abs(A[i]) @ np.abs(B[:, j]))
            worst = max(worst, float(err) / nrm)
    return worst


def test_sampled_error_is_the_exact_error():
    A = wl.random_matrix(20, 300, 2.0, 11)
    B = wl.random_matrix(300, 15, 2.0, 12)
    C = A @ B
    rows, cols = np.array([0, 5, 19]), np.array([0, 7, 14])
    got = bench.sampled_error(C, A, B, rows, cols)
    want = exact_scaled_error(C, A, B, rows, cols)
    assert abs(got - want) <= 1e-6 * want


def test_sampled_error_sees_a_one_ulp_change_and_wide_ranges():
    A = wl.random_matrix(6, 64, 4.0, 13)
    B = wl.random_matrix(64, 5, 4.0, 14)
    A[2] *= 2.0 ** 300
    A[4] *= 2.0 ** -300
    C = A @ B
    C[2, 3] = np.nextafter(C[2, 3], np.inf)
    rows, cols = np.arange(6), np.arange(5)
    got = bench.sampled_error(C, A, B, rows, cols)
    want = exact_scaled_error(C, A, B, rows, cols)
    assert abs(got - want) <= 1e-6 * want


def test_sampled_error_skips_non_finite_rows_and_exact_products_are_zero():
    A = np.array(wl.random_matrix(4, 16, 0.0, 15) * 64, order="F").round()
    B = np.array(wl.random_matrix(16, 3, 0.0, 16) * 64, order="F").round()
    C = A @ B                      # small integers: exact
    A[1, 3] = np.inf
    assert bench.sampled_error(C, A, B, np.arange(4), np.arange(3)) == 0.0


def test_sample_indices():
    assert list(bench.sample_indices(5, 8)) == [0, 1, 2, 3, 4]
    idx = bench.sample_indices(4096, 3)
    assert list(idx) == [0, 2048, 4095]
