"""The other dense configurations at their full sizes, in the launch
configuration bench.py times (oz2_dgemm_ex on a preallocated workspace with
per-stage events), checked against the oracle on what it can compute at
these sizes:

* the scan exponents and the fallback flags of every row of A and column of
  B (the oracle's scan and lower-median rule over the full operands);
* the "+1" pass: for sampled rows, max_j U_ij of the oracle's exact
  power-of-two product equals the kernel's row maximum, and the reported
  u_max is the exponent of the largest row maximum;
* the scales: s from u_max, every e_j, and d_i of the sampled rows (Eq. scale
  with reading R-scale);
* for sampled outputs, C_ij bit for bit against the correctly rounded
  X·2^-(d_i+e_j) with X = Σ_l Ã_il B̃_lj summed exactly (the value the
  residues and the CRT must reproduce, since |X| ≤ 2^T < M/2 is checked too),
  and against the oracle's FMA chain on flagged rows.

The 4096³ bench workload has its own full oracle comparison in
test_gpu_dgemm.py.
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


def run_bench_config(oz, A, B, r):
    """The bench's timed call: the library's workspace-taking entry with
    stage events, on column-major device operands."""
    import torch
    m, k = A.shape
    n = B.shape[1]
    dA, dB = to_dev(A), to_dev(B)
    C = torch.empty((n, m), dtype=torch.float64, device="cuda").t()
    ws = torch.empty(oz.oz2_workspace_size(m, n, k, r), dtype=torch.uint8, device="cuda")
    oz.oz2_dgemm_ex(dA, dB, C=C, num_moduli=r, flags=oz.FLAG_TIMING, workspace=ws)
    torch.cuda.synchronize()
    stats = oz.oz2_get_stats()
    assert oz.oz2_check_device_status() == 0
    v = {name: t.cpu().numpy() for name, t in oz.workspace_views(ws, m, n, k, r).items()
         if name in ("ra", "cb", "row_flag", "col_flag", "d", "e", "urow")}
    del dA, dB, ws
    return C, v, stats


def exact_dot(a_row, b_col):
    return sum(int(x) * int(y) for x, y in zip(a_row.tolist(), b_col.tolist()))


def check_full_size(oz, A, B, r, rows, cols):
    m, k = A.shape
    n = B.shape[1]
    mods = orc.moduli(r)
    T = orc.range_exponent(mods, "tz")
    c = orc.magnitude_clamp(k)
    C, v, stats = run_bench_config(oz, A, B, r)

    # Scan and flags over the full operands.
    ra, nfa, nza = orc.scan_rows(A)
    cb, nfb, nzb = orc.scan_rows(B.T)
    rf, _ = orc.fallback_flags(ra, nfa, nza)
    cf, _ = orc.fallback_flags(cb, nfb, nzb)
    zr, zc = rf | ~nza, cf | ~nzb
    ra, cb = np.where(zr, 0, ra), np.where(zc, 0, cb)
    assert np.array_equal((v["row_flag"] & 1).astype(bool), rf)
    assert np.array_equal((v["col_flag"] & 1).astype(bool), cf)
    assert np.array_equal(v["ra"], ra) and np.array_equal(v["cb"], cb)

    # "+1" pass and scales.
    urow = v["urow"].astype(np.float64)
    u_max = int(orc.ceil_log2_abs(urow.max())) if urow.max() > 0 else 0
    assert stats["u_max"] == u_max
    s = min(62, (T - u_max) // 2)
    assert stats["s"] == s
    assert np.array_equal(v["e"], np.where(zc, 0, s - cb))
    qb = orc.magnitude_exponents(B.T, cb, c, zc)
    qa = orc.magnitude_exponents(A[rows], ra[rows], c, zr[rows])
    U2c = orc.plus_one_pass(qa, qb.T, c)
    del qb
    for a, i in enumerate(rows):
        row_max = U2c[a].max()
        assert urow[i] * 2.0 ** (2 * c) == float(row_max)
        u_i = int(orc.ceil_log2_int(row_max)) - 2 * c if row_max > 0 else u_max
        assert v["d"][i] == (0 if zr[i] else min(62, T - s - u_i) - ra[i])

    # Sampled outputs, bit for bit.
    d, e = v["d"].astype(np.int64), v["e"].astype(np.int64)
    At = orc.quantise(np.where(zr[rows, None], 0.0, A[rows]), d[rows])
    Bt = orc.quantise(np.where(zc[cols, None], 0.0, B[:, cols].T), e[cols])
    import torch
    Crows = C.index_select(0, torch.as_tensor(rows, device=C.device)).cpu().numpy()
    for a, i in enumerate(rows):
        for b, j in enumerate(cols):
            got = Crows[a, j]
            if rf[i] or cf[j]:
                want = orc.native_entry(A, B, i, j)
            else:
                bound = exact_dot(np.abs(At[a]), np.abs(Bt[b]))
                assert bound <= 2 ** T
                want = orc.unscale_one(exact_dot(At[a], Bt[b]), -int(d[i] + e[j]))
            assert got == want and np.signbit(got) == np.signbit(want), (i, j, got, want)
    return C


def sample_cols(n, count, seed):
    rng = np.random.default_rng(seed)
    return np.unique(np.concatenate([[0, n - 1], rng.choice(n, size=count, replace=False)]))


def test_16384_cubed_r13(oz):
    """The GEMM ceiling configuration: m = n = k = 16384, φ = 1, r = 13."""
    w = wl.WORKLOADS["dgemm_16384"]
    A, B = wl.make_inputs(w)
    check_full_size(oz, A, B, w.r, rows=np.array([0, 1, 8191, w.m - 1]), cols=sample_cols(w.n, 40, 5))


def test_tall_k_full_size(oz):
    """m = n = 1024, k = 65536, φ = 0.5, r = 12."""
    w = wl.WORKLOADS["dgemm_tallk"]
    A, B = wl.make_inputs(w)
    check_full_size(oz, A, B, w.r, rows=np.array([0, 513, w.m - 1]), cols=sample_cols(w.n, 30, 6))


def test_k64_wide_full_size_with_fallback_rows(oz):
    """m = n = 16384, k = 64, φ = 4, 1% of A's rows scaled by 2^±300."""
    w = wl.WORKLOADS["dgemm_k64_wide"]
    A, B = wl.make_inputs(w)
    amax = np.abs(A).max(axis=1)
    flagged = np.flatnonzero(amax > 2.0 ** 200).tolist() + np.flatnonzero(amax < 2.0 ** -200).tolist()
    rows = np.unique(np.array([0, 1, 9000, w.m - 1] + flagged[:1] + flagged[-1:]))
    check_full_size(oz, A, B, w.r, rows=rows, cols=sample_cols(w.n, 60, 7))
