"""Parity for the character of the other dense configurations, at sizes the
oracle finishes in seconds: every entry bit-exact, with ragged shapes that
span several 256-wide tiles.

* φ = 1 at r = 13 (the 16384³ case's spread and moduli count: thirteen
  moduli take the reconstruction's five-limb path);
* k = 40000 (the tall-K case: two K-slabs for the square moduli, ten for the
  merged nonsquare ones);
* k = 64 with φ = 4 and 1% of A's rows scaled by 2^±300 (the wide case:
  native-FP64 fallback rows);
* a batched GEMV, Y = A·X with 16 right-hand sides.
"""
import numpy as np
import pytest

import workloads as wl
from helpers import ensure_built, to_dev
from oracle import cref
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


def run(oz, A, B, r):
    C, ws = oz.oz2_dgemm_ex(to_dev(A), to_dev(B), num_moduli=r)
    v = oz.workspace_views(ws, A.shape[0], B.shape[1], A.shape[1], r)
    out = {name: v[name].cpu().numpy() for name in ("d", "e", "row_flag", "col_flag")}
    out["C"] = C.cpu().numpy()
    assert oz.oz2_check_device_status() == 0
    return out


def assert_same(got, want):
    same = (got == want) | (np.isnan(got) & np.isnan(want))
    assert same.all(), f"{(~same).sum()} entries differ; first {np.argwhere(~same)[0]}"
    assert np.array_equal(np.signbit(got), np.signbit(want))


def check(got, res, rows=None):
    assert np.array_equal(got["d"], res.d) and np.array_equal(got["e"], res.e)
    assert np.array_equal((got["row_flag"] & 1).astype(bool), res.row_flag)
    assert np.array_equal((got["col_flag"] & 1).astype(bool), res.col_flag)
    assert_same(got["C"] if rows is None else got["C"][rows], res.C)


def test_phi1_r13_character(oz):
    w = wl.WORKLOADS["dgemm_16384"]
    A, B = wl.make_inputs(w, m=523, n=389, k=1601)
    res = orc.oz2_dgemm(A, B, w.r)
    got = run(oz, A, B, w.r)
    check(got, res)
    assert cref.scaled_error(got["C"], A, B, rows=np.arange(0, 523, 61)) <= 1e-15


def test_tallk_character(oz):
    w = wl.WORKLOADS["dgemm_tallk"]
    A, B = wl.make_inputs(w, m=137, n=71, k=40000)
    res = orc.oz2_dgemm(A, B, w.r)
    got = run(oz, A, B, w.r)
    check(got, res)
    assert cref.scaled_error(got["C"], A, B, rows=np.arange(0, 137, 17)) <= 1e-15


def test_k64_wide_character_with_fallback_rows(oz):
    w = wl.WORKLOADS["dgemm_k64_wide"]
    A, B = wl.make_inputs(w, m=1800, n=700)
    prep = orc.prepare(A, B, w.r)
    flagged = np.flatnonzero(prep.row_flag)
    assert len(flagged) == int(np.ceil(w.scaled_rows * 1800))     # the 2^±300 rows, and only they
    normal = np.flatnonzero(~prep.row_flag)
    # every emulated row, and one row scaled each way (the oracle's FMA chains are slow)
    rows = np.sort(np.concatenate([normal, flagged[:1], flagged[-1:]]))
    res = orc.evaluate_rows(prep, A, B, rows=rows)
    got = run(oz, A, B, w.r)
    check(got, res, rows)


def test_gemv_batch16_character(oz):
    w = wl.WORKLOADS["gemv_batch16"]
    A, B = wl.make_inputs(w, m=1500, k=2100)
    res = orc.oz2_dgemm(A, B, w.r)
    got = run(oz, A, B, w.r)
    check(got, res)
    assert cref.scaled_error(got["C"], A, B, rows=np.arange(0, 1500, 97)) <= 1e-15


def test_very_long_k_many_slabs(oz):
    """k = 262144: the residue GEMM splits K into 12 parts of 171 k-blocks,
    and each part carries its nonsquare moduli's partial residue in the
    accumulators over six 4096-entry K-slabs; the "+1" pass clamp is at its
    small end (c = 3)."""
    m, n, k = 9, 7, 262144  # one ragged tile: the slab logic is per tile
    A = np.array(wl.random_matrix(m, k, 0.5, 9300), order="F")
    B = np.array(wl.random_matrix(k, n, 0.5, 9400), order="F")
    res = orc.oz2_dgemm(A, B, 12)
    got = run(oz, A, B, 12)
    check(got, res)
    assert cref.scaled_error(got["C"], A, B, rows=np.arange(m)) <= 1e-15
