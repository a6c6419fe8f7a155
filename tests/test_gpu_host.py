"""The host-buffer entry oz2_dgemm_host against the CPU oracle, bit for bit.

The entry copies B in, then A by column chunks (four of at least 32 MB for
A of 128 MB or more), while the scan of each arrived part runs; the row keys
of A are maxima merged across its chunks.  It then runs the residue GEMM,
the reconstruction and the fallback by column blocks (oz2_plan's
host_widths) and copies each block of C back while the next one is
computed.  The result must depend on neither.
"""
import numpy as np
import pytest

import workloads as wl
from helpers import ensure_built
from oracle import ozaki2 as orc
from test_gpu_full_size import check_full_size, sample_cols

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


def pinned_colmajor(x):
    """A pinned CPU tensor holding x column-major (stride 1 down a column)."""
    import torch
    t = torch.empty((x.shape[1], x.shape[0]), dtype=torch.float64, pin_memory=True)
    t.copy_(torch.from_numpy(np.ascontiguousarray(x.T)))
    return t.t()


def assert_same(got, want):
    same = (got == want) | (np.isnan(got) & np.isnan(want))
    assert same.all(), f"{(~same).sum()} entries differ; first {np.argwhere(~same)[0]}"
    assert np.array_equal(np.signbit(got), np.signbit(want))


def test_column_blocks_with_fallback_and_padded_c(oz):
    """n = 2600: blocks of 1280 and 1320 columns.  A fallback row (2^300)
    and a zero row in A; a NaN column in each block's range and a 2^-200
    column at the end; C with leading dimension m + 5."""
    import torch
    m, n, k = 300, 2600, 70
    assert oz.oz2_plan(m, n, k, 12)["host_widths"] == [1280, 1320]
    A = np.array(wl.random_matrix(m, k, 1.0, 7100), order="F")
    B = np.array(wl.random_matrix(k, n, 1.0, 7200), order="F")
    A[7, :] *= 2.0 ** 300
    A[123, :] = 0.0
    B[3, 1500] = np.nan
    B[5, 40] = np.nan
    B[:, 2599] *= 2.0 ** -200
    want = orc.oz2_dgemm(A, B, 12).C
    C = torch.full((n, m + 5), 7.0, dtype=torch.float64, pin_memory=True).t()[:m]
    oz.oz2_dgemm_host(pinned_colmajor(A), pinned_colmajor(B), C)
    assert_same(C.numpy(), want)
    assert oz.oz2_check_device_status() == 0


def test_one_block_from_numpy(oz):
    m, n, k = 257, 300, 129
    A = np.array(wl.random_matrix(m, k, 0.5, 7300), order="F")
    B = np.array(wl.random_matrix(k, n, 0.5, 7400), order="F")
    C = oz.oz2_dgemm_host(A, B, num_moduli=9)
    assert_same(C, orc.oz2_dgemm(A, B, 9).C)


def test_empty_k_gives_zero(oz):
    m, n = 40, 1800
    A = np.zeros((m, 0), order="F")
    B = np.zeros((0, n), order="F")
    C = np.full((m, n), 3.0, order="F")
    oz.oz2_dgemm_host(A, B, C)
    assert np.array_equal(C, np.zeros((m, n))) and not np.signbit(C).any()


@pytest.mark.parametrize("seed", range(4))
def test_randomised_wide_problems(oz, seed):
    """Seeded wide problems (n from 1400 to 3400, drawn until the plan has
    at least two column blocks, the last one ragged), r from 1 to 16, φ from
    0 to 5, and planted special rows of A and columns of B in random
    blocks."""
    rng = np.random.default_rng(8000 + seed)
    for _ in range(100):
        m = int(rng.integers(150, 500))
        n = int(rng.integers(1400, 3400))
        k = int(rng.integers(1, 120))
        r = int(rng.integers(1, 17))
        if len(oz.oz2_plan(m, n, k, r)["host_widths"]) >= 2:
            break
    assert len(oz.oz2_plan(m, n, k, r)["host_widths"]) >= 2
    phi = float(rng.uniform(0.0, 5.0))
    A = np.array(wl.random_matrix(m, k, phi, 8100 + seed), order="F")
    B = np.array(wl.random_matrix(k, n, phi, 8200 + seed), order="F")
    for _ in range(int(rng.integers(0, 3))):
        i = int(rng.integers(0, m))
        A[i, :] *= 2.0 ** (300 if rng.integers(0, 2) else -300)
    for _ in range(int(rng.integers(0, 4))):
        j, kind = int(rng.integers(0, n)), int(rng.integers(0, 3))
        if kind == 0:
            B[:, j] = 0.0
        elif kind == 1:
            B[int(rng.integers(0, k)), j] = np.inf
        else:
            B[:, j] *= 2.0 ** -250
    want = orc.oz2_dgemm(A, B, r).C
    got = oz.oz2_dgemm_host(A, B, num_moduli=r)
    assert_same(got, want)
    assert oz.oz2_check_device_status() == 0


def test_column_blocks_with_split_k(oz):
    """A short C with a long k: each column block's residue GEMM splits k
    (blocks of 1536 and 1064 columns in 2 and 5 parts on a GB300), with a
    fallback row and a zero column.  C equals the device-buffer entry's bit
    for bit, whose sampled outputs, scales and flags are checked against the
    oracle."""
    m, n, k = 128, 2600, 20000
    plan = oz.oz2_plan(m, n, k, 12)
    assert plan["host_widths"] == [1536, 1064] and min(plan["host_kparts"][:2]) > 1
    A = np.array(wl.random_matrix(m, k, 1.0, 7500), order="F")
    B = np.array(wl.random_matrix(k, n, 1.0, 7600), order="F")
    A[9, :] *= 2.0 ** -300
    B[:, 2000] = 0.0
    want = check_full_size(oz, A, B, 12, rows=np.array([0, 9, 64, 127]), cols=sample_cols(n, 30, 8))
    got = oz.oz2_dgemm_host(A, B, num_moduli=12)
    assert_same(got, want.cpu().numpy())
    assert oz.oz2_check_device_status() == 0


@pytest.mark.parametrize("pad", [0, 3])
def test_operand_chunks_merge_scans(oz, pad):
    """A of 128 MB arrives in four column chunks (pitched copies when its
    leading dimension is m + pad).  Row 5's largest entry and row 77's
    outlier (2^400, a fallback row) lie in later chunks, row 300 holds a NaN
    in the second; column 7 of B is 2^-300 (a fallback column).  C equals
    the device-buffer entry's bit for bit, whose flags, exponents, scales
    and sampled outputs are checked against the oracle."""
    import torch
    m, n, k = 2048, 512, 8192
    A = np.array(wl.random_matrix(m, k, 0.5, 7700), order="F")
    B = np.array(wl.random_matrix(k, n, 0.5, 7800), order="F")
    A[5, 7000] = 2.0 ** 40
    A[77, 5000] = 2.0 ** 400
    A[300, 3000] = np.nan
    B[:, 7] *= 2.0 ** -300
    rows = np.array([0, 5, 77, 1024, m - 1])  # row 300 (NaN) is compared with the device entry only
    want = check_full_size(oz, A, B, 12, rows=rows, cols=np.unique(np.concatenate([[7], sample_cols(n, 24, 9)])))
    hA = A
    if pad:
        hA = torch.full((k, m + pad), 5.0, dtype=torch.float64, pin_memory=True).t()[:m]
        hA.copy_(torch.from_numpy(A))
        assert hA.stride() == (1, m + pad)
    got = oz.oz2_dgemm_host(hA, B, num_moduli=12)
    assert_same(got, want.cpu().numpy())
    st = oz.oz2_get_stats()
    assert st["fallback_rows"] == 2 and st["fallback_cols"] == 1
    assert oz.oz2_check_device_status() == 0
