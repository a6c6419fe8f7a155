"""Pin the oracle's scaling, residue products, Garner and unscale to
mathematics that does not come from the oracle itself: brute-force exact
integer products, the CRT round trip, closed-form bounds, textbook special
cases, and planted mistakes that must be caught."""
import math
import random
from fractions import Fraction

import numpy as np
import pytest

import workloads as wl
from oracle import cref
from oracle import ozaki2 as oz


def small_inputs(m, n, k, phi=0.5, seed=7):
    A = wl.random_matrix(m, k, phi, seed)
    B = wl.random_matrix(k, n, phi, seed + 1)
    return A, B


# ------------------------------------------------------------------ Garner
@pytest.mark.parametrize("r", [1, 2, 3, 5, 12, 13, 16])
def test_crt_round_trip(r):
    mods = oz.moduli(r)
    M = oz.modulus_product(mods)
    rng = random.Random(r)
    xs = [-(M // 2), M - M // 2 - 1, 0, 1, -1] + [rng.randrange(-(M // 2), M - M // 2) for _ in range(300)]
    res = np.array([[int(oz.centred(x % m, m)) for x in xs] for m in mods], dtype=np.int64)
    X = oz.garner_value(res, mods)
    assert [int(v) for v in X] == xs


def test_garner_digits_are_mixed_radix():
    """v_k ∈ [0, m_k) and Σ v_k P_{k-1} ≡ C^(i) (mod m_i) (App. A)."""
    mods = oz.moduli(12)
    rng = np.random.default_rng(3)
    res = np.stack([oz.centred(rng.integers(0, m, 50), m) for m in mods])
    v = oz.garner_digits(res, mods)
    for k, m in enumerate(mods):
        assert (v[k] >= 0).all() and (v[k] < m).all()
    X = oz.garner_value(res, mods)
    for i, m in enumerate(mods):
        assert all(int(x) % m == int(c) % m for x, c in zip(X, res[i]))


def test_mutation_garner_dropped_term_is_caught(monkeypatch):
    mods = oz.moduli(4)
    xs = list(range(-500000, 500000, 99991))
    res = np.array([[int(oz.centred(x % m, m)) for x in xs] for m in mods], dtype=np.int64)

    def bad_digits(res, mods):
        v = []
        for k, mk in enumerate(mods):
            acc = res[k] % mk
            P = 1
            for j in range(k - 1):          # planted: drops the last term
                acc = (acc - v[j] * (P % mk)) % mk
                P *= mods[j]
            for j in range(max(k - 1, 0), k):
                P *= mods[j]
            inv = pow(P % mk, -1, mk) if k else 1
            v.append((acc * inv) % mk)
        return v

    monkeypatch.setattr(oz, "garner_digits", bad_digits)
    X = oz.garner_value(res, mods)
    assert [int(v) for v in X] != xs


# ------------------------------------------------- brute force, tiny inputs
@pytest.mark.parametrize("quant", ["tz", "rn"])
@pytest.mark.parametrize("scale", ["r2", "r1"])
@pytest.mark.parametrize("shape", [(1, 1, 1), (3, 5, 7), (8, 8, 33), (17, 9, 64)])
def test_brute_force_exact_integer_product(shape, scale, quant):
    m, n, k = shape
    A, B = small_inputs(m, n, k, phi=1.0, seed=sum(shape))
    res = oz.oz2_dgemm(A, B, 12, quant=quant, scale=scale)
    # Eq. (M-bound): the range bound and the exactness of the CRT value
    At = [[int(x) for x in row] for row in res.At]
    Bt = [[int(x) for x in row] for row in res.Bt]
    M = oz.modulus_product(res.mods)
    for i in range(m):
        for j in range(n):
            exact = sum(At[i][l] * Bt[l][j] for l in range(k))
            absum = sum(abs(At[i][l] * Bt[l][j]) for l in range(k))
            T_tz = oz.range_exponent(res.mods, "tz")
            assert absum <= 2**T_tz < M / 2
            assert int(res.X[i, j]) == exact
            for idx, mi in enumerate(res.mods):
                assert int(res.residues[idx, i, j]) == int(oz.centred(exact % mi, mi))
            want = float(Fraction(exact) * Fraction(2) ** (-int(res.d[i]) - int(res.e[j])))
            assert res.C[i, j] == want
    # quantiser definition: |Ã| ≤ 2^62 and the rule itself
    for i in range(m):
        for l in range(k):
            y = Fraction(float(A[i, l])) * Fraction(2) ** int(res.d[i])
            q = int(y) if quant == "tz" else round(y)   # Python round: half to even
            assert At[i][l] == q and abs(q) <= 2**62


def test_r2_scale_is_valid_and_maximal():
    """R-scale: 2^(t_i+s) U_ij ≤ 2^T and one more bit on t_i would break it."""
    A, B = small_inputs(40, 30, 50, phi=2.0, seed=11)
    res = oz.oz2_dgemm(A, B, 12)
    c = res.c
    U = res.U2c.astype(object)
    t = res.d + res.ra
    for i in range(40):
        assert t[i] <= 62
        umax = max(int(x) for x in U[i])
        assert Fraction(2) ** (int(t[i]) + res.s) * Fraction(umax, 2 ** (2 * c)) <= 2 ** res.T
        if t[i] < 62:
            assert Fraction(2) ** (int(t[i]) + 1 + res.s) * Fraction(umax, 2 ** (2 * c)) > 2 ** res.T
    # and U bounds |A||B| (the "+1" pass is an upper estimate)
    for i in range(0, 40, 7):
        for j in range(0, 30, 5):
            tot = sum(Fraction(abs(float(A[i, l]))) * Fraction(abs(float(B[l, j]))) for l in range(50))
            assert tot <= Fraction(2) ** int(res.ra[i] + res.cb[j]) * Fraction(int(U[i, j]), 2 ** (2 * c))


def test_plus_one_pass_is_fp32_exact():
    for k in (1, 2, 63, 64, 65, 4096, 65536):
        c = oz.magnitude_clamp(k)
        assert 0 <= c <= 9
        assert k * 4**c <= 2**24


# ------------------------------------------------------- special cases
def test_zero_matrix():
    A = np.zeros((5, 6))
    B = wl.random_matrix(6, 4, 0.5, 1)
    res = oz.oz2_dgemm(A, B, 12)
    assert np.all(res.C == 0) and not np.signbit(res.C).any()


def test_integer_inputs_give_the_exact_product():
    rng = np.random.default_rng(5)
    A = rng.integers(-1000, 1000, size=(12, 20)).astype(np.float64)
    B = rng.integers(-1000, 1000, size=(20, 9)).astype(np.float64)
    for r in (8, 12, 16):
        res = oz.oz2_dgemm(A, B, r)
        assert np.array_equal(res.C, A @ B)


def test_single_nonzero_per_row_is_exact():
    rng = np.random.default_rng(6)
    m, k, n = 10, 12, 7
    A = np.zeros((m, k))
    for i in range(m):
        A[i, rng.integers(0, k)] = np.ldexp(float(rng.integers(1, 2**30)), int(rng.integers(-40, 40)))
    B = np.ldexp(rng.integers(-2**30, 2**30, size=(k, n)).astype(np.float64), -20)
    res = oz.oz2_dgemm(A, B, 12)
    assert np.array_equal(res.C, A @ B)


def test_truncation_bound_holds():
    A, B = small_inputs(24, 20, 48, phi=1.5, seed=21)
    for quant in ("tz", "rn"):
        for r in (6, 9, 12):
            res = oz.oz2_dgemm(A, B, r, quant=quant)
            bound = oz.truncation_bound(A, B, res.d, res.e, quant)
            for i in range(24):
                for j in range(20):
                    ex = cref.exact_entry(A[i], B[:, j])
                    err = abs(Fraction(float(res.C[i, j])) - ex)
                    assert err <= Fraction(float(bound[i, j])) * (1 + 2**-40) + abs(ex) * Fraction(2) ** -53


def test_error_target_at_r12_on_the_small_workload():
    A, B = wl.make_inputs(wl.WORKLOADS["dgemm_256"], 128, 128, 256)
    res = oz.oz2_dgemm(A, B, 12)
    assert cref.scaled_error(res.C, A, B) <= 1e-15
    res13 = oz.oz2_dgemm(A, B, 13)
    assert cref.scaled_error(res13.C, A, B) <= 1e-16


def test_error_falls_with_r():
    A, B = small_inputs(32, 32, 64)
    errs = [cref.scaled_error(oz.oz2_dgemm(A, B, r).C, A, B) for r in range(4, 13)]
    for a, b in zip(errs, errs[1:]):
        assert b < a


# ------------------------------------------------------------ unscale
def test_unscale_is_correctly_rounded():
    rng = random.Random(9)
    cases = [(2**53 + 1, 0), (2**53 + 3, 0), (-(2**53 + 1), 0), (1, -1074), (1, -1075), (3, -1076),
             (2**60 + 2**7, -1100), (2**110 - 1, 914), (2**110 - 1, 915), (5, -1077)]
    for _ in range(500):
        x = rng.randrange(-2**111, 2**111)
        cases.append((x, rng.randrange(-1200, 900)))
    for X, E in cases:
        ex = Fraction(X) * Fraction(2) ** E
        try:
            want = float(ex)
        except OverflowError:
            want = math.copysign(math.inf, X)
        got = oz.unscale_one(X, E)
        assert got == want
        if X != 0:
            assert math.copysign(1, got) == math.copysign(1, want)


# ------------------------------------------------------------ fallback
def test_fma_against_two_product():
    rng = random.Random(4)
    for _ in range(300):
        a = rng.uniform(-1, 1) * 2.0 ** rng.randrange(-60, 60)
        b = rng.uniform(-1, 1) * 2.0 ** rng.randrange(-60, 60)
        p = a * b
        # Dekker's TwoProduct gives the exact rounding error of a·b
        _, err = cref._two_product(np.float64(a), np.float64(b))
        assert oz.fma(a, b, -p) == float(err)
    assert oz.fma(math.inf, 0.0, 1.0) != oz.fma(math.inf, 0.0, 1.0)   # NaN
    assert oz.fma(2.0, 3.0, math.inf) == math.inf
    assert oz.fma(1e308, 10.0, -math.inf) == -math.inf


def test_fallback_flags_and_rows():
    A, B = small_inputs(40, 12, 16, seed=31)
    A = np.asfortranarray(A.copy())
    A[3, :] *= 2.0 ** 300
    A[7, :] *= 2.0 ** -300
    A[11, 5] = np.nan
    A[13, 2] = np.inf
    A[20, :] = 0.0
    B = np.asfortranarray(B.copy())
    B[4, 6] = -np.inf
    res = oz.oz2_dgemm(A, B, 12)
    assert list(np.flatnonzero(res.row_flag)) == [3, 7, 11, 13]
    assert list(np.flatnonzero(res.col_flag)) == [6]
    for i in (3, 7, 11, 13):
        for j in range(12):
            got, want = res.C[i, j], oz.native_entry(A, B, i, j)
            assert got == want or (np.isnan(got) and np.isnan(want))
    assert np.isnan(res.C[11]).all()
    assert np.all(res.C[20, [j for j in range(12) if j != 6]] == 0.0)
    # scaled rows are accurate: the native chain's error is ≤ k·u·|A||B|
    for i in (3, 7):
        hi, lo = cref.dot2(A[i:i + 1], B[:, :6])
        assert np.all(np.abs((res.C[i, :6] - hi[0]) - lo[0]) <= 16 * 2**-53 * (np.abs(A[i]) @ np.abs(B[:, :6])))
    # unflagged rows match the same call with the flagged rows zeroed
    A0 = A.copy()
    A0[[3, 7, 11, 13]] = 0.0
    B0 = B.copy()
    B0[:, 6] = 0.0
    ref = oz.oz2_dgemm(A0, B0, 12)
    keep = [i for i in range(40) if i not in (3, 7, 11, 13)]
    cols = [j for j in range(12) if j != 6]
    assert np.array_equal(res.C[np.ix_(keep, cols)], ref.C[np.ix_(keep, cols)])


def test_fallback_median_rule():
    e = np.array([0, 1, 2, 3, 200, -200, 129, 131, -128])
    nz = np.ones(e.size, bool)
    nz[0] = False
    flags, med = oz.fallback_flags(e, np.zeros(e.size, bool), nz)
    s = np.sort(e[nz])
    assert med == s[(s.size - 1) // 2]
    assert list(np.flatnonzero(flags)) == [i for i in range(e.size) if nz[i] and abs(e[i] - med) > 128]


# ------------------------------------------------------------ references
def test_dot2_against_exact():
    A, B = small_inputs(6, 5, 200, phi=3.0, seed=41)
    hi, lo = cref.dot2(A, B)
    for i in range(6):
        for j in range(5):
            ex = cref.exact_entry(A[i], B[:, j])
            diff = abs(Fraction(float(hi[i, j])) + Fraction(float(lo[i, j])) - ex)
            nrm = sum(Fraction(abs(float(a))) * Fraction(abs(float(b))) for a, b in zip(A[i], B[:, j]))
            assert diff <= nrm * Fraction(2) ** -90


def test_exact_entry_definition():
    rng = random.Random(2)
    a = [rng.uniform(-1, 1) * 2.0 ** rng.randrange(-30, 30) for _ in range(20)]
    b = [rng.uniform(-1, 1) * 2.0 ** rng.randrange(-30, 30) for _ in range(20)]
    assert cref.exact_entry(a, b) == sum(Fraction(x) * Fraction(y) for x, y in zip(a, b))
