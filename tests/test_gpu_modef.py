"""On-the-fly residues (A's digit planes formed on chip inside the residue
GEMM) for a skinny C, bit for bit against the oracle and against the path
that stores A's planes (the default; OZ2_FLAG_ON_THE_FLY selects the former).

The cases span one and two TMEM passes (n ≤ 16 holds every modulus's
accumulators at once; n ≤ 32 holds eight, the modulus blocking of Eq. nblk),
one to three K-slabs (residues carried in TMEM every 4096 k-entries), ragged
rows and k, every moduli count class, both quantisers and scale rules,
fallback, zero and non-finite rows, and the full 16384 × 16 × 16384
batched-GEMV workload on sampled rows.
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


def run(oz, A, B, r, flags=0, quant="tz", scale="r2"):
    import torch
    torch.cuda.synchronize()
    oz.oz2_get_stats()
    C, ws = oz.oz2_dgemm_ex(to_dev(A), to_dev(B), num_moduli=r, flags=flags, quant=quant, scale=scale)
    v = oz.workspace_views(ws, A.shape[0], B.shape[1], A.shape[1], r)
    res = v["residues"].cpu().numpy()
    launches = oz.oz2_get_stats()["kernel_launches"]
    assert oz.oz2_check_device_status() == 0
    return C.cpu().numpy(), res, launches


@pytest.mark.parametrize("shape,r", [
    ((128, 16, 1000), 12),    # one K-slab, every modulus resident
    ((300, 5, 4096), 12),     # ragged rows, exactly one slab
    ((257, 17, 5000), 12),    # two TMEM passes (8 + 4 moduli), two slabs
    ((130, 32, 9000), 16),    # two passes of eight, three slabs
    ((200, 1, 2000), 6),      # squares only
    ((150, 12, 1100), 13),    # thirteen moduli, ragged k
])
def test_on_the_fly_matches_oracle_and_stored_planes(oz, shape, r):
    m, n, k = shape
    A = np.array(wl.random_matrix(m, k, 1.0, 8000 + m + k), order="F")
    B = np.array(wl.random_matrix(k, n, 1.0, 8100 + n), order="F")
    want = orc.oz2_dgemm(A, B, r)
    C, res, launches = run(oz, A, B, r, flags=oz.FLAG_ON_THE_FLY)
    assert_same(C, want.C)
    assert np.array_equal(res, want.residues)
    C2, res2, launches2 = run(oz, A, B, r)
    assert_same(C2, want.C)
    assert np.array_equal(res2, res)
    # B-only deconstruction + the on-the-fly GEMM in place of both (which
    # never splits k); the stored-plane path adds a fold where it splits k.
    # Both add the row maxima of a split "+1" GEMM.
    plan = oz.oz2_plan(m, n, k, r, 76)
    assert launches == 11 + (plan["mag_kparts"] > 1)
    assert launches2 == 11 + (plan["mag_kparts"] > 1) + (plan["kparts"] > 1)


@pytest.mark.parametrize("quant,scale", [("rn", "r2"), ("tz", "r1"), ("rn", "r1")])
def test_variants_and_special_rows(oz, quant, scale):
    m, n, k = 260, 9, 3000
    A = np.array(wl.random_matrix(m, k, 2.0, 8201), order="F")
    B = np.array(wl.random_matrix(k, n, 2.0, 8202), order="F")
    A[3, :] *= 2.0 ** 300
    A[4, :] *= 2.0 ** -300
    A[10, :] = 0.0
    A[11, 5] = np.nan
    A[12, 7] = np.inf
    A[30, 100] = 5e-320
    A[31, :] = 3e-310        # a row whose largest entry is subnormal
    B[:, 2] = 0.0
    want = orc.oz2_dgemm(A, B, 12, quant=quant, scale=scale).C
    C, _, _ = run(oz, A, B, 12, flags=oz.FLAG_ON_THE_FLY, quant=quant, scale=scale)
    assert_same(C, want)


def test_full_batched_gemv_workload_sampled_rows(oz):
    w = wl.WORKLOADS["gemv_batch16"]
    A, B = wl.make_inputs(w)
    C, _ = oz.oz2_dgemm_ex(to_dev(A), to_dev(B), num_moduli=w.r, flags=oz.FLAG_ON_THE_FLY)
    C = C.cpu().numpy()
    assert oz.oz2_check_device_status() == 0
    rows = np.array([0, 1, 127, 128, 8191, w.m - 1])
    want = orc.oz2_dgemm(A, B, w.r, rows=rows).C
    assert_same(C[rows], want)
