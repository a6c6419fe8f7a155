"""Stage-by-stage parity of the CUDA path against the CPU oracle.

Every comparison is bit-exact: exponents, flags, E4M3 plane bytes, residue
matrices C^(i), and the FP64 results of Garner/unscale and of the native
fallback.  Inputs are seeded; shapes span several 128-tiles plus ragged tails.
"""
import numpy as np
import pytest

import workloads as wl
from helpers import ensure_built, planes_from_residues, to_dev
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


def special_inputs(m, n, k, seed):
    A = np.array(wl.random_matrix(m, k, 1.0, seed), order="F")
    B = np.array(wl.random_matrix(k, n, 1.0, seed + 1), order="F")
    A[3 % m, :] *= 2.0 ** 300
    A[5 % m, :] *= 2.0 ** -300
    A[7 % m, 1 % k] = np.nan
    A[9 % m, :] = 0.0
    A[11 % m, :] *= 2.0 ** -1000                      # subnormal-range entries
    A[13 % m, 0] = 5e-324
    B[:, 2 % n] = 0.0
    B[0, 4 % n] = np.inf
    return A, B


def oracle_flags(X):
    e, nonfinite, nonzero = orc.scan_rows(X)
    fb, _ = orc.fallback_flags(e, nonfinite, nonzero)
    zero = fb | ~nonzero
    return np.where(zero, 0, e), fb.astype(np.uint8) | (zero.astype(np.uint8) << 1)


@pytest.mark.parametrize("shape", [(40, 30, 50), (300, 260, 1100)])
def test_scan(oz, shape):
    m, n, k = shape
    A, B = special_inputs(m, n, k, 17)
    ra, cb, rf, cf = oz.oz2_scan(to_dev(A), to_dev(B))
    want_ra, want_rf = oracle_flags(A)
    want_cb, want_cf = oracle_flags(B.T)
    assert np.array_equal(ra.cpu().numpy(), want_ra)
    assert np.array_equal(rf.cpu().numpy(), want_rf)
    assert np.array_equal(cb.cpu().numpy(), want_cb)
    assert np.array_equal(cf.cpu().numpy(), want_cf)


@pytest.mark.parametrize("scale", ["r2", "r1"])
@pytest.mark.parametrize("quant", ["tz", "rn"])
@pytest.mark.parametrize("shape,r", [((40, 30, 50), 12), ((300, 260, 1100), 12), ((129, 257, 64), 16)])
def test_scale(oz, shape, r, quant, scale):
    m, n, k = shape
    A, B = special_inputs(m, n, k, 23)
    res = orc.oz2_dgemm(A, B, r, quant=quant, scale=scale, rows=[0])
    dA, dB = to_dev(A), to_dev(B)
    ra, cb, rf, cf = oz.oz2_scan(dA, dB)
    mag_a, mag_b, urow, d, e = oz.oz2_scale(dA, dB, ra, cb, rf, cf, num_moduli=r, quant=quant, scale=scale)
    assert np.array_equal(d.cpu().numpy(), res.d)
    assert np.array_equal(e.cpu().numpy(), res.e)
    if scale == "r2":
        k_pad = (k + 127) // 128 * 128
        enc = np.vectorize(lambda q: 0 if q < -10**5 else orc.e4m3_encode_power_of_two(int(q)), otypes=[np.uint8])
        want_a = np.zeros((m, k_pad), np.uint8)
        want_a[:, :k] = enc(res.qa)
        want_b = np.zeros((n, k_pad), np.uint8)
        want_b[:, :k] = enc(res.qb)
        assert np.array_equal(mag_a.cpu().numpy(), want_a)
        assert np.array_equal(mag_b.cpu().numpy(), want_b)
        want_u = (res.U2c.max(axis=1) / 4.0 ** res.c).astype(np.float32)
        assert np.array_equal(urow.cpu().numpy(), want_u)


@pytest.mark.parametrize("quant", ["tz", "rn"])
@pytest.mark.parametrize("shape,r", [((40, 30, 50), 12), ((200, 136, 300), 12), ((70, 65, 130), 16),
                                     ((33, 17, 1), 1), ((64, 64, 256), 5)])
def test_deconstruct(oz, shape, r, quant):
    m, n, k = shape
    A, B = special_inputs(m, n, k, 29)
    res = orc.oz2_dgemm(A, B, r, quant=quant, rows=[0])
    dA, dB = to_dev(A), to_dev(B)
    _, _, rf, cf = oz.oz2_scan(dA, dB)
    import torch
    d = torch.from_numpy(res.d.astype(np.int32)).cuda()
    e = torch.from_numpy(res.e.astype(np.int32)).cuda()
    pa, pb = oz.oz2_deconstruct(dA, dB, d, e, rf, cf, num_moduli=r, quant=quant)
    k_pad = (k + 127) // 128 * 128
    mods = orc.moduli(r)
    want_a = planes_from_residues([orc.centred(res.At, mi) for mi in mods], mods, orc, k_pad, merged=True)
    want_b = planes_from_residues([orc.centred(res.Bt.T, mi) for mi in mods], mods, orc, k_pad)
    assert np.array_equal(pa.cpu().numpy(), want_a)
    assert np.array_equal(pb.cpu().numpy(), want_b)


def _residue_case(oz, m, n, k, r, gen, simt=False):
    mods = orc.moduli(r)
    k_pad = (k + 127) // 128 * 128
    a = [gen(mi, (m, k), 0) for mi in mods]
    b = [gen(mi, (n, k), 1) for mi in mods]
    pa = planes_from_residues(a, mods, orc, k_pad, merged=True)   # A: last nonsquare plane is -16·d1
    pb = planes_from_residues(b, mods, orc, k_pad)
    import torch
    got = oz.oz2_residue_gemm(torch.from_numpy(pa).cuda(), torch.from_numpy(pb).cuda(), m, n, k, r, simt=simt)
    got = got.cpu().numpy()
    for i, mi in enumerate(mods):
        h = mi - mi // 2
        want = orc.centred(orc.exact_int_matmul(a[i], b[i].T, h, h), mi)
        assert np.array_equal(got[i], want), f"modulus {mi}"


def _uniform(seed):
    rng = np.random.default_rng(seed)
    return lambda mi, shape, side: orc.centred(rng.integers(0, mi, size=shape), mi)


@pytest.mark.parametrize("simt", [False, True])
@pytest.mark.parametrize("shape,r", [((128, 128, 128), 12), ((200, 136, 300), 12), ((384, 256, 1024), 12),
                                     ((130, 70, 260), 16), ((1, 1, 1), 3)])
def test_residue_gemm_uniform(oz, shape, r, simt):
    _residue_case(oz, *shape, r, _uniform(sum(shape) + r), simt=simt)


def test_residue_gemm_k_slabs(oz):
    """k above the K-slabs (32768 for squares, 4096 for nonsquare moduli): the
    epilogue folds the slabs mod m."""
    _residue_case(oz, 128, 136, 33000, 4, _uniform(5))
    _residue_case(oz, 300, 260, 9000, 8, _uniform(6))


def _merged_argmax(m):
    """Centred residues (d, e) maximising |d0e0 - 16 d1e1| for a nonsquare m."""
    d = np.arange(-(m // 2), m - m // 2)
    d0, d1 = orc.nonsquare_digits(d)
    t = np.abs(d0[:, None] * d0[None, :] - 16 * d1[:, None] * d1[None, :])
    i, j = np.unravel_index(np.argmax(t), t.shape)
    return int(d[i]), int(d[j]), int(t[i, j])


def test_residue_gemm_merged_accumulator_worst_case(oz):
    """The merged nonsquare accumulator at its bound: 4096 terms of 4095
    (Eq. accum-exact with K_slab = 4096), then a second slab."""
    mods = orc.moduli(12)

    def gen(mi, shape, side):
        rows, kk = shape
        if orc.square_base(mi):
            return np.full(shape, mi // 2, dtype=np.int64)
        d, e, t = _merged_argmax(mi)
        assert t >= 3900
        out = np.full(shape, d if side == 0 else e, dtype=np.int64)
        out[1::2, 4096:] = -out[1::2, 4096:]
        return out

    _residue_case(oz, 256, 256, 8192, 12, gen)


def test_residue_gemm_accumulator_extremes(oz):
    """Accumulators reach 2^24 exactly (Eq. accum-exact at K_slab = 32768), and
    small products follow large partial sums (a truncating accumulator fails)."""
    k = 32768

    def extreme(mi, shape, side):
        rows, kk = shape
        out = np.empty(shape, dtype=np.int64)
        top = mi // 2                                  # 544 for 1089: digits (16, 16)
        out[:, : kk // 2] = top
        out[:, kk // 2:] = 1
        out[1::2, kk // 2:] = -1                       # cancellation in odd rows
        return out

    _residue_case(oz, 128, 128, k, 1, extreme)          # modulus 1089 alone
    _residue_case(oz, 128, 128, k, 8, extreme)          # squares and two nonsquares


def test_reconstruct(oz):
    import torch
    rng = np.random.default_rng(41)
    cases = [(r, 70, 33, None) for r in (1, 2, 7, 12, 13, 16)]
    cases += [(12, 71, 5, 74), (12, 71, 6, 75), (13, 9, 7, 9), (5, 1, 3, 1)]  # odd rows, odd/even ld
    for r, m, n, ldr in cases:
        mods = orc.moduli(r)
        R = np.stack([orc.centred(rng.integers(0, mi, size=(m, n)), mi) for mi in mods])
        R[:, 0, 0] = 0
        d = rng.integers(40, 80, size=m)
        e = rng.integers(40, 80, size=n)
        if m > 3:
            d[1], d[2], d[3] = 1100, 1180, -1100            # subnormal, underflow, overflow rows
        if ldr is None:
            res = torch.from_numpy(np.ascontiguousarray(R).astype(np.int16)).cuda()
        else:   # column-major storage with the given leading dimension
            buf = torch.full((r, n, ldr), 777, dtype=torch.int16)
            buf[:, :, :m] = torch.from_numpy(R.transpose(0, 2, 1).astype(np.int16))
            res = buf.cuda()[:, :, :m].transpose(1, 2)
            assert res.stride() == (n * ldr, 1, ldr)
        C = oz.oz2_reconstruct(res, torch.from_numpy(d.astype(np.int32)).cuda(),
                               torch.from_numpy(e.astype(np.int32)).cuda(), m, n, r).cpu().numpy()
        X = orc.garner_value(R, mods)
        for i in range(m):
            for j in range(n):
                want = orc.unscale_one(int(X[i, j]), -int(d[i]) - int(e[j]))
                assert C[i, j] == want and np.signbit(C[i, j]) == np.signbit(want), (r, m, n, i, j)


@pytest.mark.parametrize("r,m,n,ldr,ldc,c_off", [
    (12, 1100, 5, 1104, 1100, 0),    # several row blocks, the last ragged
    (12, 1031, 4, 1040, 1032, 0),    # odd m: the last row runs in the element-wise kernel
    (16, 600, 3, 608, 600, 0),       # five-limb path
    (6, 8, 1, 8, 8, 0),              # one short column
    (11, 300, 4, 304, 300, 1),       # C not 16-byte aligned: element-wise kernel
    (12, 64, 3, 64, 65, 0),          # odd ldc: element-wise kernel
])
def test_reconstruct_tiles_and_alignment(oz, r, m, n, ldr, ldc, c_off):
    """The row-pair kernel on ragged row blocks and an odd last row, and the
    element-wise kernel for buffers the row-pair one cannot take, against
    Garner's algorithm in the oracle; rows of C beyond m stay untouched."""
    import torch
    rng = np.random.default_rng(1000 + m)
    mods = orc.moduli(r)
    R = np.stack([orc.centred(rng.integers(0, mi, size=(m, n)), mi) for mi in mods])
    R[:, :7, 0] = 0                                    # X = 0 for a few outputs
    d = rng.integers(40, 80, size=m)
    e = rng.integers(40, 80, size=n)
    d[1], d[2], d[3] = 1100, 1180, -1100               # subnormal, underflow, overflow rows
    buf = torch.full((r, n, ldr), 777, dtype=torch.int16)
    buf[:, :, :m] = torch.from_numpy(R.transpose(0, 2, 1).astype(np.int16))
    res = buf.cuda()[:, :, :m].transpose(1, 2)
    cbuf = torch.full((n * ldc + c_off,), 12345.0, dtype=torch.float64, device="cuda")
    C = cbuf[c_off:].view(n, ldc).t()[:m, :]
    oz.oz2_reconstruct(res, torch.from_numpy(d.astype(np.int32)).cuda(), torch.from_numpy(e.astype(np.int32)).cuda(),
                       m, n, r, C=C)
    got = C.cpu().numpy()
    X = orc.garner_value(R, mods)
    for i in range(m):
        for j in range(n):
            want = orc.unscale_one(int(X[i, j]), -int(d[i]) - int(e[j]))
            assert got[i, j] == want and np.signbit(got[i, j]) == np.signbit(want), (r, m, n, i, j)
    # rows beyond m of each column of C are untouched
    full = cbuf[c_off:].view(n, ldc).cpu().numpy()
    assert (full[:, m:] == 12345.0).all()


def test_reconstruct_many_outputs_left_to_the_exact_path(oz):
    """Two rows and more columns than the launch has column strides, so each
    thread walks about ten columns, with most outputs within M/2^13 of ±M/2,
    which the fast path leaves to Garner's algorithm: threads leave more
    outputs than their list holds and find the rest again by rescanning;
    small, zero and other outputs are mixed in."""
    import random
    import torch
    r = 12
    mods = orc.moduli(r)
    M = orc.modulus_product(mods)
    rng = random.Random(77)
    m, n = 2, 12500
    xs = []
    lo, hi, band = -(M // 2), M - M // 2 - 1, M >> 13
    for _ in range(m * n):
        t = rng.random()
        if t < 0.35:
            xs.append(lo + rng.randrange(band))
        elif t < 0.7:
            xs.append(hi - rng.randrange(band))
        elif t < 0.8:
            xs.append(0)
        elif t < 0.9:
            xs.append(rng.randrange(-(1 << 80), 1 << 80))
        else:
            xs.append(rng.randrange(-(M // 4), M // 4))
    X = np.array(xs, dtype=object).reshape(m, n)
    R = np.zeros((r, m, n), dtype=np.int64)
    for k, mk in enumerate(mods):
        R[k] = np.vectorize(lambda x: int(orc.centred(x % mk, mk)), otypes=[np.int64])(X)
    d = np.array([3, -40], dtype=np.int64)
    e = np.array([rng.randrange(-60, 60) for _ in range(n)], dtype=np.int64)
    C = oz.oz2_reconstruct(torch.from_numpy(R.astype(np.int16)).cuda(), torch.from_numpy(d.astype(np.int32)).cuda(),
                           torch.from_numpy(e.astype(np.int32)).cuda(), m, n, r).cpu().numpy()
    for i in range(m):
        for j in range(n):
            want = orc.unscale_one(int(X[i, j]), -int(d[i]) - int(e[j]))
            assert C[i, j] == want and np.signbit(C[i, j]) == np.signbit(want), (i, j)


def test_reconstruct_near_the_range_boundary(oz):
    """Integers at and next to ±M/2, where the fast reconstruction defers to
    Garner's algorithm, and a band of values around them."""
    import random
    import torch
    for r in (3, 12, 13, 16):
        mods = orc.moduli(r)
        M = orc.modulus_product(mods)
        lo, hi = -(M // 2), M - M // 2 - 1
        rng = random.Random(r)
        xs = [lo, lo + 1, hi, hi - 1, 0, 1, -1]
        band = max(1, M >> 13)
        xs += [lo + rng.randrange(band) for _ in range(60)] + [hi - rng.randrange(band) for _ in range(60)]
        # Either side of the fast path's margin (X within M/2^12 of ±M/2).
        edge = M >> 12
        xs += [lo + edge + rng.randrange(-band, band) for _ in range(40)]
        xs += [hi - edge + rng.randrange(-band, band) for _ in range(40)]
        xs += [rng.randrange(lo, hi + 1) for _ in range(60)]
        m, n = len(xs), 3
        R = np.zeros((r, m, n), dtype=np.int64)
        for i, x in enumerate(xs):
            for k, mk in enumerate(mods):
                R[k, i, :] = int(orc.centred(x % mk, mk))
        d = np.full(m, 5, dtype=np.int64)
        e = np.array([0, 40, -1100], dtype=np.int64)
        res = torch.from_numpy(R.astype(np.int16)).cuda()
        C = oz.oz2_reconstruct(res, torch.from_numpy(d.astype(np.int32)).cuda(),
                               torch.from_numpy(e.astype(np.int32)).cuda(), m, n, r).cpu().numpy()
        for i, x in enumerate(xs):
            for j in range(n):
                want = orc.unscale_one(x, -int(d[i]) - int(e[j]))
                assert C[i, j] == want and np.signbit(C[i, j]) == np.signbit(want), (r, i, j)


def test_reconstruct_next_to_rounding_midpoints(oz):
    """Integers X placed at and around the midpoints between doubles of
    X·2^E, at several bit lengths, where the fixed-point fast path must
    defer to an exact path unless its estimate decides the rounding."""
    import random
    import torch
    for r in (9, 11, 12):
        mods = orc.moduli(r)
        M = orc.modulus_product(mods)
        rng = random.Random(100 + r)
        xs = []
        for b in range(max(60, M.bit_length() - 40), M.bit_length() - 1, 3):
            q = b - 53
            for off in (0, 1, -1, 1 << 20, -(1 << 20), 1 << 30, -(1 << 30), 1 << 34, -(1 << 34), 1 << 36):
                if off and abs(off) >= 1 << (q - 1):
                    continue
                x = (rng.randrange(1 << 52, 1 << 53) << q) + (1 << (q - 1)) + off
                if x < M // 2:
                    xs.append(x * rng.choice((1, -1)))
        xs += [rng.randrange(-(M // 2), M // 2) for _ in range(40)]
        m, n = len(xs), 2
        R = np.zeros((r, m, n), dtype=np.int64)
        for i, x in enumerate(xs):
            for k, mk in enumerate(mods):
                R[k, i, :] = int(orc.centred(x % mk, mk))
        d = np.full(m, 3, dtype=np.int64)
        e = np.array([-M.bit_length(), 60], dtype=np.int64)
        res = torch.from_numpy(R.astype(np.int16)).cuda()
        C = oz.oz2_reconstruct(res, torch.from_numpy(d.astype(np.int32)).cuda(),
                               torch.from_numpy(e.astype(np.int32)).cuda(), m, n, r).cpu().numpy()
        for i, x in enumerate(xs):
            for j in range(n):
                want = orc.unscale_one(x, -int(d[i]) - int(e[j]))
                assert C[i, j] == want and np.signbit(C[i, j]) == np.signbit(want), (r, i, j)


def test_reconstruct_other_representatives(oz):
    """Residues in (-m_i, m_i) that are not the centred ones give the same
    results as the centred ones (the reconstruction's input contract)."""
    import torch
    rng = np.random.default_rng(43)
    for r in (5, 12, 13):
        mods = orc.moduli(r)
        m, n = 40, 36
        R = np.stack([orc.centred(rng.integers(0, mi, size=(m, n)), mi) for mi in mods])
        shift = rng.integers(0, 2, size=R.shape).astype(bool)
        Ralt = R.copy()
        for k, mk in enumerate(mods):
            moved = np.where(R[k] < 0, R[k] + mk, np.where(R[k] > 0, R[k] - mk, 0))
            Ralt[k] = np.where(shift[k], moved, R[k])
            assert (np.abs(Ralt[k]) < mk).all()
        d = rng.integers(40, 80, size=m)
        e = rng.integers(40, 80, size=n)
        dev_d = torch.from_numpy(d.astype(np.int32)).cuda()
        dev_e = torch.from_numpy(e.astype(np.int32)).cuda()
        C1 = oz.oz2_reconstruct(torch.from_numpy(R.astype(np.int16)).cuda(), dev_d, dev_e, m, n, r).cpu().numpy()
        C2 = oz.oz2_reconstruct(torch.from_numpy(Ralt.astype(np.int16)).cuda(), dev_d, dev_e, m, n, r).cpu().numpy()
        X = orc.garner_value(R, mods)
        for i in range(m):
            for j in range(n):
                want = orc.unscale_one(int(X[i, j]), -int(d[i]) - int(e[j]))
                assert C1[i, j] == want and C2[i, j] == want, (r, i, j)


def test_fallback_rows_and_columns(oz):
    import torch
    m, n, k = 70, 60, 50
    A, B = special_inputs(m, n, k, 53)
    rf = np.zeros(m, np.uint8)
    cf = np.zeros(n, np.uint8)
    rows, cols = [3, 5, 7, 40, 69], [4, 11, 59]
    rf[rows] = 1
    cf[cols] = 1
    C0 = np.full((m, n), 7.0)
    C = to_dev(C0)
    oz.oz2_fallback(to_dev(A), to_dev(B), torch.from_numpy(rf).cuda(), torch.from_numpy(cf).cuda(), C)
    got = C.cpu().numpy()
    for i in range(m):
        for j in range(n):
            if i in rows or j in cols:
                want = orc.native_entry(A, B, i, j)
                assert got[i, j] == want or (np.isnan(got[i, j]) and np.isnan(want))
            else:
                assert got[i, j] == 7.0


def test_native_dgemm(oz):
    A = wl.random_matrix(37, 53, 0.5, 3)
    B = wl.random_matrix(53, 29, 0.5, 4)
    got = oz.oz2_native_dgemm(to_dev(A), to_dev(B)).cpu().numpy()
    for i in range(0, 37, 5):
        for j in range(0, 29, 4):
            assert got[i, j] == orc.native_entry(A, B, i, j)
