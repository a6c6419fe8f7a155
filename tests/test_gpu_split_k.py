"""Split K in the residue GEMM, bit for bit against the oracle.

A problem with few output tiles and a long k fills few waves of the CTA
pairs, so the residue GEMM runs each unit's k-blocks in parts and sums the
parts' residues mod m (Eq. modgemm is a sum over k).  Each case checks the
scales, every residue matrix C^(i) and C against the oracle, and that the
call did split: it launches one kernel more (the fold) than an unsplit call,
besides the row-maximum kernel of a split "+1" magnitude GEMM where the
plan reports one (mag_kparts).
"""
import numpy as np
import pytest

import workloads as wl
from helpers import ensure_built, to_dev
from oracle import ozaki2 as orc

pytestmark = pytest.mark.gpu



def unsplit_launches(oz, m, n, k, r):
    """Kernels of a call whose residue GEMM does not split: prepare, 2 scan
    (A and B in one launch, then the flags), magnitude, "+1", scales,
    deconstruct, GEMM, CRT, 2 fallback, and the row maxima of a split "+1"
    GEMM.  (C here has ld = m: for even m the CRT takes every row in pairs,
    for odd m it runs the element-wise instance alone, so it is one launch
    either way.)"""
    return 11 + (oz.oz2_plan(m, n, k, r, 76)["mag_kparts"] > 1)


@pytest.fixture(scope="module")
def oz():
    ensure_built()
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2606_06510_gb300 as oz
    oz.lib()
    return oz


def run_counted(oz, A, B, r):
    """C, the workspace views and the number of kernels the call launched."""
    import torch
    dA, dB = to_dev(A), to_dev(B)
    torch.cuda.synchronize()
    oz.oz2_get_stats()  # resets the launch counter
    C, ws = oz.oz2_dgemm_ex(dA, dB, num_moduli=r)
    torch.cuda.synchronize()
    launches = oz.oz2_get_stats()["kernel_launches"]
    v = oz.workspace_views(ws, A.shape[0], B.shape[1], A.shape[1], r)
    assert oz.oz2_check_device_status() == 0
    return C.cpu().numpy(), {k: v[k].cpu().numpy() for k in ("d", "e", "residues")}, launches


def check(oz, A, B, r, split):
    want = orc.oz2_dgemm(A, B, r)
    C, v, launches = run_counted(oz, A, B, r)
    assert launches == unsplit_launches(oz, A.shape[0], B.shape[1], A.shape[1], r) + (1 if split else 0)
    assert np.array_equal(v["d"], want.d) and np.array_equal(v["e"], want.e)
    assert np.array_equal(v["residues"], want.residues)
    same = (C == want.C) | (np.isnan(C) & np.isnan(want.C))
    assert same.all(), f"{(~same).sum()} entries differ; first {np.argwhere(~same)[0]}"
    num = ~np.isnan(C)  # a NaN's sign is not part of the result
    assert np.array_equal(np.signbit(C[num]), np.signbit(want.C[num]))


@pytest.mark.parametrize("shape,r", [
    ((200, 150, 20000), 12),   # one tile, parts of 27 k-blocks (nonsquare slabs carried inside)
    ((64, 64, 3000), 16),      # five-limb reconstruction, parts of 8 k-blocks
    ((300, 40, 9000), 6),      # square moduli only, two tile rows
    ((9, 7, 70000), 12),       # ragged tile, ragged last part
    ((3, 5, 1000), 12),        # the shortest parts (4 k-blocks: short slabs)
])
def test_split_k_bit_exact(oz, shape, r):
    m, n, k = shape
    A = np.array(wl.random_matrix(m, k, 1.0, 9500 + m), order="F")
    B = np.array(wl.random_matrix(k, n, 1.0, 9600 + n), order="F")
    check(oz, A, B, r, split=True)


def test_split_k_square_slabs_inside_parts(oz):
    """Parts of 261 k-blocks: longer than a square modulus's 32768-entry
    K-slab, so the square accumulators carry their residue inside a part."""
    m, n, k = 520, 260, 100000
    A = np.array(wl.random_matrix(m, k, 0.5, 9700), order="F")
    B = np.array(wl.random_matrix(k, n, 0.5, 9800), order="F")
    check(oz, A, B, 4, split=True)


def test_split_k_with_fallback_rows_and_zero_columns(oz):
    m, n, k = 100, 90, 12000
    A = np.array(wl.random_matrix(m, k, 1.0, 9900), order="F")
    B = np.array(wl.random_matrix(k, n, 1.0, 9901), order="F")
    A[5, :] *= 2.0 ** 300
    A[17, 100] = np.inf
    B[:, 33] = 0.0
    B[:, 60] *= 2.0 ** -250
    check(oz, A, B, 12, split=True)


def test_many_tiles_do_not_split(oz):
    """1536 × 1280 outputs (30 tiles × 12 moduli = 360 units, over four
    waves of the 76 CTA pairs): no split, whatever k."""
    m, n, k = 1536, 1280, 1536
    A = np.array(wl.random_matrix(m, k, 0.5, 9950), order="F")
    B = np.array(wl.random_matrix(k, n, 0.5, 9951), order="F")
    C, _, launches = run_counted(oz, A, B, 12)
    assert oz.oz2_plan(m, n, k, 12, 76)["kparts"] == 1
    assert launches == unsplit_launches(oz, m, n, k, 12)
    rows = np.arange(0, m, 97)
    want = orc.oz2_dgemm(A, B, 12, rows=rows)
    assert np.array_equal(C[rows], want.C)
