"""oz2_dgemm_noalloc: the emulated DGEMM for callers that cannot allocate
device memory (their framework's allocator owns it, or an allocation may not
block or fail at run time).  It runs in a fixed 32 MiB scratch array inside
the library instead of a workspace, so its results must match oz2_dgemm's
exactly, call after call, even though every call reuses the same scratch.

This file is collected last on purpose: it exercises process-wide device
state (the scratch array) and must pass both alone and after the other tests.
"""
import ctypes

import numpy as np
import pytest

import workloads as wl
from helpers import ensure_built, to_dev
from oracle import ozaki2 as orc

pytestmark = pytest.mark.gpu

LIMIT = 32 << 20


@pytest.fixture(scope="module")
def env():
    ensure_built()
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2606_06510_gb300 as oz
    raw = ctypes.CDLL(oz.LIB_PATH)
    f = raw.oz2_dgemm_noalloc
    I64, P = ctypes.c_int64, ctypes.c_void_p
    f.restype = ctypes.c_int
    f.argtypes = [I64, I64, I64, P, I64, P, I64, P, I64, ctypes.c_int, P]
    return oz, f, torch


def call_noalloc(env, A, B, r):
    oz, f, torch = env
    m, k = A.shape
    n = B.shape[1]
    C = torch.full((n, m), np.nan, dtype=torch.float64, device="cuda").t()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    rc = f(m, n, k, ctypes.c_void_p(A.data_ptr()), m, ctypes.c_void_p(B.data_ptr()), k,
           ctypes.c_void_p(C.data_ptr()), m, r, stream)
    assert rc == 0, oz.oz2_status_string(rc)
    torch.cuda.synchronize()
    assert oz.oz2_check_device_status() == 0
    return C.cpu().numpy()


@pytest.mark.parametrize("r", [12, 16])
def test_matches_oz2_dgemm_on_consecutive_calls(env, r):
    oz, _, _ = env
    shapes = [(256, 256, 256, 0.5), (200, 136, 300, 2.0)]   # second call: other shape, other data
    for idx, (m, n, k, phi) in enumerate(shapes):
        assert oz.oz2_workspace_size(m, n, k, r) <= LIMIT
        A = to_dev(wl.random_matrix(m, k, phi, 100 * r + idx))
        B = to_dev(wl.random_matrix(k, n, phi, 100 * r + idx + 50))
        got = call_noalloc(env, A, B, r)
        want = oz.oz2_dgemm(A, B, num_moduli=r).cpu().numpy()
        # bit-identical: same kernels, same arithmetic
        assert np.array_equal(got, want)


def test_rejects_problems_beyond_the_scratch(env):
    oz, f, _ = env
    m = n = k = 1024
    assert oz.oz2_workspace_size(m, n, k, 12) > LIMIT
    rc = f(m, n, k, None, m, None, k, None, m, 12, None)   # rejected before any device work
    assert rc == -6          # OZ2_ERR_UNSUPPORTED


def test_matches_the_oracle(env):
    """One call checked directly against the oracle (not only against
    oz2_dgemm), bit for bit, with a fallback row and a zero column."""
    m, n, k, r = 200, 136, 300, 12
    A = np.array(wl.random_matrix(m, k, 1.0, 4242), order="F")
    B = np.array(wl.random_matrix(k, n, 1.0, 4243), order="F")
    A[7, :] *= 2.0 ** 300
    B[:, 40] = 0.0
    got = call_noalloc(env, to_dev(A), to_dev(B), r)
    want = orc.oz2_dgemm(A, B, r).C
    same = (got == want) | (np.isnan(got) & np.isnan(want))
    assert same.all(), f"{(~same).sum()} entries differ from the oracle"


@pytest.mark.parametrize("shape,r,parts", [((64, 64, 3000), 12, 4), ((128, 64, 2500), 14, 2)])
def test_split_k_in_the_scratch_then_an_unsplit_call(env, shape, r, parts):
    """A small C with a long k: the residue GEMM splits k and keeps the
    parts' residues in the scratch array's magnitude-plane region.  The
    split call (two launches more than an unsplit one: the fold, and the row
    maxima of the "+1" GEMM, which splits k as well) must match
    oz2_dgemm bit for bit, and an unsplit call right after it must too."""
    oz, _, _ = env
    m, n, k = shape
    assert oz.oz2_workspace_size(m, n, k, r) <= LIMIT
    assert oz.oz2_plan(m, n, k, r, 76)["kparts"] == parts
    A = to_dev(wl.random_matrix(m, k, 1.0, 5151 + r))
    B = to_dev(wl.random_matrix(k, n, 1.0, 5252 + r))
    assert oz.oz2_plan(m, n, k, r, 76)["mag_kparts"] > 1  # the "+1" GEMM splits k too
    oz.oz2_get_stats()                      # resets the launch counter
    got = call_noalloc(env, A, B, r)
    assert oz.oz2_get_stats()["kernel_launches"] == 13
    want = oz.oz2_dgemm(A, B, num_moduli=r).cpu().numpy()
    assert np.array_equal(got, want)
    A2 = to_dev(wl.random_matrix(96, 300, 0.5, 5353 + r))
    B2 = to_dev(wl.random_matrix(300, 80, 0.5, 5454 + r))
    assert oz.oz2_plan(96, 80, 300, r, 76)["mag_kparts"] == 1
    oz.oz2_get_stats()
    got2 = call_noalloc(env, A2, B2, r)
    assert oz.oz2_get_stats()["kernel_launches"] == 11
    assert np.array_equal(got2, oz.oz2_dgemm(A2, B2, num_moduli=r).cpu().numpy())
