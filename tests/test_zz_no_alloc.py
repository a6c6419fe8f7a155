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
