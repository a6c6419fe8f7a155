"""The fused residue GEMM + reconstruction (OZ2_FLAG_FUSED; r = 11, 12,
k ≤ 256), bit for bit against the oracle and against the two-launch path.

The fused kernel keeps each output's residues on chip and folds them into
the reconstruction's 96-bit fixed-point sum; outputs whose rounding that sum
cannot decide go to a list and are recomputed exactly.  The cases span
ragged tiles (128 rows × 32 columns), one and two k-blocks, fallback and
zero rows and columns, non-finite entries, outputs that are exactly zero
without a zero row or column (they all take the list), and the full
16384 × 16384 × 64 wide-range workload on sampled rows.
"""
import numpy as np
import pytest

import workloads as wl
from helpers import ensure_built, to_dev
from oracle import ozaki2 as orc

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def oz():
    ensure_built()
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2606_06510_gb300 as oz
    oz.lib()
    return oz


def assert_same(got, want):
    same = (got == want) | (np.isnan(got) & np.isnan(want))
    if not same.all():
        bad = np.argwhere(~same)
        i, j = bad[0]
        raise AssertionError(f"{len(bad)} entries differ; first ({i},{j}): {got[i, j]!r} vs {want[i, j]!r}")
    num = ~np.isnan(got)
    assert np.array_equal(np.signbit(got[num]), np.signbit(want[num]))


def run(oz, A, B, r, flags=0):
    import torch
    torch.cuda.synchronize()
    oz.oz2_get_stats()
    C, _ = oz.oz2_dgemm_ex(to_dev(A), to_dev(B), num_moduli=r, flags=flags)
    C = C.cpu().numpy()
    launches = oz.oz2_get_stats()["kernel_launches"]
    assert oz.oz2_check_device_status() == 0
    return C, launches


@pytest.mark.parametrize("r", [11, 12])
@pytest.mark.parametrize("shape", [(300, 77, 64), (129, 33, 1), (1, 1, 100), (64, 500, 128), (257, 95, 200),
                                   (130, 64, 256)])
def test_fused_matches_oracle_and_unfused(oz, shape, r):
    m, n, k = shape
    A = np.array(wl.random_matrix(m, k, 2.0, 7000 + m + k), order="F")
    B = np.array(wl.random_matrix(k, n, 2.0, 7100 + n), order="F")
    want = orc.oz2_dgemm(A, B, r).C
    C, launches = run(oz, A, B, r, flags=oz.FLAG_FUSED)
    assert_same(C, want)
    C2, launches2 = run(oz, A, B, r)
    assert_same(C2, want)
    assert launches == launches2 == 11   # fused GEMM + list pass in place of GEMM + reconstruction


def test_fallback_zero_and_non_finite_rows_and_columns(oz):
    m, n, k = 200, 150, 64
    A = np.array(wl.random_matrix(m, k, 4.0, 7201), order="F")
    B = np.array(wl.random_matrix(k, n, 4.0, 7202), order="F")
    A[3, :] *= 2.0 ** 300
    A[4, :] *= 2.0 ** -300
    A[10, :] = 0.0
    A[11, 5] = np.nan
    A[12, 7] = np.inf
    B[:, 20] = 0.0
    B[:, 21] *= 2.0 ** 280
    B[9, 22] = -np.inf
    A[30, 1] = 5e-320    # subnormal entries
    B[2, 40] = -3e-310
    want = orc.oz2_dgemm(A, B, 12).C
    C, _ = run(oz, A, B, 12, flags=oz.FLAG_FUSED)
    assert_same(C, want)


def test_exactly_zero_outputs_take_the_exact_path(oz):
    """Rows and columns with nonzero entries whose products cancel exactly:
    X = 0 there, which the fixed-point estimate cannot round, so every such
    output goes through the list and its exact reconstruction (+0)."""
    m, n, k = 96, 70, 64
    rng = np.random.default_rng(7300)
    A = np.asfortranarray(rng.integers(-8, 9, size=(m, k)).astype(np.float64))
    B = np.asfortranarray(rng.integers(-8, 9, size=(k, n)).astype(np.float64))
    A[:, 1::2] = A[:, 0::2]          # column pairs of A equal ...
    B[1::2, :40] = -B[0::2, :40]     # ... against row pairs of B that cancel: C[:, :40] = 0
    A[5, :] += 1.0
    want = orc.oz2_dgemm(A, B, 12).C
    assert (want[:, :40][np.arange(m) != 5] == 0).all()
    C, _ = run(oz, A, B, 12, flags=oz.FLAG_FUSED)
    assert_same(C, want)


def test_full_wide_range_workload_sampled_rows(oz):
    w = wl.WORKLOADS["dgemm_k64_wide"]
    A, B = wl.make_inputs(w)
    C, _ = oz.oz2_dgemm_ex(to_dev(A), to_dev(B), num_moduli=w.r, flags=oz.FLAG_FUSED)
    C = C.cpu().numpy()
    assert oz.oz2_check_device_status() == 0
    big = np.flatnonzero(np.abs(A).max(axis=1) > 2.0 ** 200)
    rows = np.unique(np.concatenate([[0, 1, 8191, w.m - 1], big[:2]]))
    want = orc.oz2_dgemm(A, B, w.r, rows=rows).C
    assert_same(C[rows], want)
