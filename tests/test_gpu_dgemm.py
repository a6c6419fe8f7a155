"""End-to-end parity of oz2_dgemm / oz2_dgemm_ex with the CPU oracle.

Small and ragged shapes compare every entry bit-for-bit, along with the
intermediates left in the workspace.  The 4096³ workload that bench.py times
is checked in the same launch configuration: full scale vectors and a
sample of rows of C, bit-exact.
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


def run_ex(oz, A, B, r, quant="tz", scale="r2", flags=0):
    C, ws = oz.oz2_dgemm_ex(to_dev(A), to_dev(B), num_moduli=r, quant=quant, scale=scale, flags=flags)
    views = oz.workspace_views(ws, A.shape[0], B.shape[1], A.shape[1], r)
    assert oz.oz2_check_device_status() == 0
    return C.cpu().numpy(), {k: v.cpu().numpy() for k, v in views.items()}


def assert_same(got, want):
    same = (got == want) | (np.isnan(got) & np.isnan(want))
    if not same.all():
        bad = np.argwhere(~same)
        i, j = bad[0]
        raise AssertionError(f"{len(bad)} entries differ; first ({i},{j}): {got[i, j]!r} vs {want[i, j]!r}")
    assert np.array_equal(np.signbit(got[~np.isnan(got)]), np.signbit(want[~np.isnan(want)]))


def test_small_workload_bit_exact_and_accurate(oz):
    A, B = wl.make_inputs(wl.WORKLOADS["dgemm_256"])
    res = orc.oz2_dgemm(A, B, 12)
    C, v = run_ex(oz, A, B, 12)
    assert_same(C, res.C)
    assert np.array_equal(v["d"], res.d) and np.array_equal(v["e"], res.e)
    assert np.array_equal(v["residues"], res.residues)
    assert cref.scaled_error(C, A, B) <= 1e-15
    # the production entry (own workspace) gives the same bits, and so does
    # the fused residue GEMM and reconstruction
    C2 = oz.oz2_dgemm(to_dev(A), to_dev(B), num_moduli=12).cpu().numpy()
    assert_same(C2, res.C)
    C3, _ = run_ex(oz, A, B, 12, flags=oz.FLAG_FUSED)
    assert_same(C3, res.C)


@pytest.mark.parametrize("shape", [(1, 1, 1), (100, 77, 333), (257, 129, 129), (64, 300, 7), (3, 5, 1000)])
def test_ragged_shapes(oz, shape):
    m, n, k = shape
    A = wl.random_matrix(m, k, 1.0, m + n)
    B = wl.random_matrix(k, n, 1.0, k)
    res = orc.oz2_dgemm(A, B, 12)
    C, _ = run_ex(oz, A, B, 12)
    assert_same(C, res.C)


@pytest.mark.parametrize("r", [1, 2, 6, 11, 12, 13, 16])
def test_moduli_counts(oz, r):
    A, B = wl.random_matrix(64, 160, 0.5, 1), wl.random_matrix(160, 48, 0.5, 2)
    res = orc.oz2_dgemm(A, B, r)
    C, v = run_ex(oz, A, B, r)
    assert_same(C, res.C)
    assert np.array_equal(v["residues"], res.residues)
    C, _ = run_ex(oz, A, B, r, flags=oz.FLAG_FUSED)   # fused for r = 11, 12 (k = 160)
    assert_same(C, res.C)


@pytest.mark.parametrize("quant", ["tz", "rn"])
@pytest.mark.parametrize("scale", ["r2", "r1"])
def test_variants(oz, quant, scale):
    A, B = wl.random_matrix(96, 200, 2.0, 5), wl.random_matrix(200, 80, 2.0, 6)
    res = orc.oz2_dgemm(A, B, 12, quant=quant, scale=scale)
    C, _ = run_ex(oz, A, B, 12, quant=quant, scale=scale)
    assert_same(C, res.C)


def test_simt_diagnostic_engine_matches(oz):
    A, B = wl.random_matrix(130, 140, 1.0, 8), wl.random_matrix(140, 70, 1.0, 9)
    res = orc.oz2_dgemm(A, B, 12)
    C, _ = run_ex(oz, A, B, 12, flags=oz.FLAG_DEBUG_SIMT_GEMM)
    assert_same(C, res.C)


def test_fallback_and_special_values(oz):
    A = np.array(wl.random_matrix(150, 90, 1.0, 11), order="F")
    B = np.array(wl.random_matrix(90, 70, 1.0, 12), order="F")
    A[3, :] *= 2.0 ** 300
    A[8, :] *= 2.0 ** -300
    A[20, 4] = np.nan
    A[21, 5] = -np.inf
    A[30, :] = 0.0
    A[31, :] *= 2.0 ** -1060
    B[7, 9] = np.inf
    B[:, 12] = 0.0
    res = orc.oz2_dgemm(A, B, 12)
    C, v = run_ex(oz, A, B, 12)
    assert_same(C, res.C)
    st = oz.oz2_get_stats()
    # rows 3, 8 (2^±300), 20, 21 (non-finite) and 31 (2^-1060: far below the median)
    assert st["fallback_rows"] == int(res.row_flag.sum()) == 5
    assert st["fallback_cols"] == int(res.col_flag.sum()) == 1
    assert np.array_equal(v["row_flag"] & 1, res.row_flag.astype(np.uint8))


def test_zero_and_empty(oz):
    import torch
    A = np.zeros((50, 40))
    B = wl.random_matrix(40, 30, 0.5, 1)
    C, _ = run_ex(oz, A, B, 12)
    assert np.all(C == 0) and not np.signbit(C).any()
    # k = 0: C = 0
    Cd = to_dev(np.full((5, 6), 3.0))
    oz.oz2_dgemm(torch.empty((5, 0), dtype=torch.float64, device="cuda"),
                 torch.empty((0, 6), dtype=torch.float64, device="cuda"), C=Cd)
    assert np.all(Cd.cpu().numpy() == 0)


def test_integer_inputs_exact(oz):
    rng = np.random.default_rng(3)
    A = rng.integers(-2**20, 2**20, size=(70, 90)).astype(np.float64)
    B = rng.integers(-2**20, 2**20, size=(90, 50)).astype(np.float64)
    C, _ = run_ex(oz, A, B, 12)
    assert np.array_equal(C, A @ B)


@pytest.mark.parametrize("quant", ["tz", "rn"])
def test_subnormal_rows(oz, quant):
    """Rows of A whose entries are all subnormal: no row is out of range of
    the others, so none falls back, and their scales exceed 1083 (the
    deconstruction's general quantisation path).  A normal row and a zero
    row sit beside them."""
    m, n, k = 70, 90, 130
    A = np.array(wl.random_matrix(m, k, 0.5, 9100), order="F") * 2.0 ** -1060
    A[5, :] = np.array(wl.random_matrix(1, k, 0.5, 9101))[0] * 2.0 ** -1000   # normal, 60 binades up
    A[9, :] = 0.0
    assert np.abs(A[10]).max() < 2.2250738585072014e-308 and np.abs(A[10]).max() > 0
    B = np.array(wl.random_matrix(k, n, 0.5, 9200), order="F")
    res = orc.oz2_dgemm(A, B, 12, quant=quant)
    C, v = run_ex(oz, A, B, 12, quant=quant)
    assert v["d"].max() > 1083
    assert np.array_equal(v["d"], res.d) and np.array_equal(v["e"], res.e)
    assert_same(C, res.C)


def test_bench_workload_full_size_sampled(oz):
    """4096³, r = 12, φ = 0.5: the configuration bench.py times."""
    w = wl.WORKLOADS["dgemm_4096"]
    A, B = wl.make_inputs(w)
    rows = np.array([0, 1, 127, 128, 2048, 4000, 4095])
    res = orc.oz2_dgemm(A, B, w.r, rows=rows)
    C, v = run_ex(oz, A, B, w.r)
    assert np.array_equal(v["d"], res.d) and np.array_equal(v["e"], res.e)
    assert_same(C[rows], res.C)
    assert cref.scaled_error(C, A, B, rows=rows[:3]) <= 1e-15


def test_cuda_graph_capture_and_replay(oz):
    """The production calls are stream-ordered end to end (pool allocation,
    memsets, launches), so they can be captured into a CUDA graph; replays
    on new input values in the same buffers give the direct call's bits."""
    import torch
    A1, B1 = wl.make_inputs(wl.WORKLOADS["dgemm_256"], m=300, n=200, k=333)
    A2, B2 = wl.random_matrix(300, 333, 1.0, 77), wl.random_matrix(333, 200, 1.0, 78)
    dA, dB = to_dev(A1), to_dev(B1)
    C = torch.empty((200, 300), dtype=torch.float64, device="cuda").t()
    ws = torch.empty(oz.oz2_workspace_size(300, 200, 333, 12), dtype=torch.uint8, device="cuda")
    s = torch.cuda.Stream()
    for call in ("dgemm", "dgemm_ex"):
        run = (lambda: oz.oz2_dgemm(dA, dB, C=C, num_moduli=12, stream=s)) if call == "dgemm" else \
              (lambda: oz.oz2_dgemm_ex(dA, dB, C=C, num_moduli=12, workspace=ws, stream=s))
        with torch.cuda.stream(s):
            run()                                   # warm-up outside the capture (device set-up)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            run()
        for A, B in ((A2, B2), (A1, B1)):
            dA.copy_(to_dev(A))
            dB.copy_(to_dev(B))
            g.replay()
            torch.cuda.synchronize()
            want = oz.oz2_dgemm(to_dev(A), to_dev(B), num_moduli=12).cpu().numpy()
            assert_same(C.cpu().numpy(), want)
        assert oz.oz2_check_device_status() == 0


@pytest.mark.parametrize("pad", [(3, 5, 7), (1, 0, 2), (8, 8, 8)])
def test_leading_dimensions_larger_than_rows(oz, pad):
    """A, B and C as sub-matrix views of larger column-major arrays (lda > m,
    ldb > k, ldc > m, odd and even paddings): the same bits as contiguous
    operands, and C's padding rows are left untouched."""
    import torch
    m, n, k = 261, 133, 299
    A, B = wl.make_inputs(wl.WORKLOADS["dgemm_256"], m=m, n=n, k=k)
    res = orc.oz2_dgemm(A, B, 12)
    pa, pb, pc = pad
    bigA = torch.full((k, m + pa), 7.0, dtype=torch.float64, device="cuda")
    bigB = torch.full((n, k + pb), -3.0, dtype=torch.float64, device="cuda")
    bigC = torch.full((n, m + pc), 11.0, dtype=torch.float64, device="cuda")
    dA = bigA.t()[:m, :]
    dB = bigB.t()[:k, :]
    dC = bigC.t()[:m, :]
    dA.copy_(torch.from_numpy(np.ascontiguousarray(A)).cuda())
    dB.copy_(torch.from_numpy(np.ascontiguousarray(B)).cuda())
    assert dA.stride() == (1, m + pa) and dB.stride() == (1, k + pb) and dC.stride() == (1, m + pc)
    oz.oz2_dgemm(dA, dB, C=dC, num_moduli=12)
    assert_same(dC.cpu().numpy(), res.C)
    if pc:
        assert (bigC.t()[m:, :] == 11.0).all()
    assert oz.oz2_check_device_status() == 0


def test_concurrent_calls_on_two_streams(oz):
    """Two different problems issued back to back on two streams (each call
    with its own workspace from the library pool) give their own results."""
    import torch
    A1, B1 = wl.make_inputs(wl.WORKLOADS["dgemm_256"], m=300, n=270, k=260)
    A2, B2 = wl.random_matrix(200, 500, 1.0, 91), wl.random_matrix(500, 180, 1.0, 92)
    want1, want2 = orc.oz2_dgemm(A1, B1, 12).C, orc.oz2_dgemm(A2, B2, 13).C
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    d = [to_dev(x) for x in (A1, B1, A2, B2)]
    torch.cuda.synchronize()
    for _ in range(3):
        C1 = oz.oz2_dgemm(d[0], d[1], num_moduli=12, stream=s1)
        C2 = oz.oz2_dgemm(d[2], d[3], num_moduli=13, stream=s2)
        torch.cuda.synchronize()
        assert_same(C1.cpu().numpy(), want1)
        assert_same(C2.cpu().numpy(), want2)
    assert oz.oz2_check_device_status() == 0


def test_wait_expiry_is_reported_and_the_context_stays_usable(oz):
    """The failure path of every bounded wait, without a GPU fault: a wait
    that nothing completes expires after ~1 ms, the host reads
    OZ2_ERR_TIMEOUT once, and the next emulated DGEMM is exact."""
    import torch
    assert oz.oz2_check_device_status() == 0
    oz.oz2_selftest_timeout(2_000_000)
    torch.cuda.synchronize()
    assert oz.oz2_check_device_status() == -5         # OZ2_ERR_TIMEOUT
    assert oz.oz2_check_device_status() == 0          # read once, then cleared
    A, B = wl.make_inputs(wl.WORKLOADS["dgemm_256"], m=130, n=70, k=90)
    C = oz.oz2_dgemm(to_dev(A), to_dev(B), num_moduli=12).cpu().numpy()
    assert_same(C, orc.oz2_dgemm(A, B, 12).C)
    assert oz.oz2_check_device_status() == 0


@pytest.mark.parametrize("seed", range(12))
def test_randomised_problems_bit_exact(oz, seed):
    """Seeded random problems: shapes 1..300, exponent spread φ ∈ [0, 6],
    r ∈ [1, 16], every quantiser/scale variant, and planted special rows and
    columns (zeros, 2^±300 scaling, subnormal entries, an Inf or NaN).  Every
    entry of C, d and e bit-exact against the oracle."""
    rng = np.random.default_rng(4000 + seed)
    m, n, k = (int(v) for v in rng.integers(1, 301, size=3))
    phi = float(rng.uniform(0.0, 6.0))
    r = int(rng.integers(1, 17))
    quant = ("tz", "rn")[seed % 2]
    scale = ("r2", "r1")[(seed // 2) % 2] if seed % 3 else "r2"
    A = np.array(wl.random_matrix(m, k, phi, 5000 + seed), order="F")
    B = np.array(wl.random_matrix(k, n, phi, 6000 + seed), order="F")
    for _ in range(int(rng.integers(0, 4))):           # planted rows of A
        i, kind = int(rng.integers(0, m)), int(rng.integers(0, 5))
        if kind == 0:
            A[i, :] = 0.0
        elif kind == 1:
            A[i, :] *= 2.0 ** 300
        elif kind == 2:
            A[i, :] *= 2.0 ** -300
        elif kind == 3:
            A[i, int(rng.integers(0, k))] = 5e-324 * int(rng.integers(1, 1000))
        else:
            A[i, int(rng.integers(0, k))] = (np.inf, -np.inf, np.nan)[int(rng.integers(0, 3))]
    for _ in range(int(rng.integers(0, 3))):           # planted columns of B
        j, kind = int(rng.integers(0, n)), int(rng.integers(0, 3))
        if kind == 0:
            B[:, j] = 0.0
        elif kind == 1:
            B[:, j] *= 2.0 ** -200
        else:
            B[int(rng.integers(0, k)), j] = np.nan
    res = orc.oz2_dgemm(A, B, r, quant=quant, scale=scale)
    C, v = run_ex(oz, A, B, r, quant=quant, scale=scale)
    assert np.array_equal(v["d"], res.d) and np.array_equal(v["e"], res.e)
    assert_same(C, res.C)
