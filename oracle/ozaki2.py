"""Plain, slow, exact CPU oracle for Ozaki Scheme II DGEMM on FP8 digit planes.

TEST INFRASTRUCTURE ONLY -- never imported by the product path.

Every function follows one passage of the paper (arxiv 2606.06510, "FP8 is
All You Need (Part 1)") and is written to be checked against it by eye:

* §2.3 "Ozaki Scheme II", Phase 1, Eq. (scale): power-of-two diagonals D, E
  and the integer matrices  Ã = ⌊DA⌉,  B̃ = ⌊BE⌉  (quantiser TZ or RN,
  Table "numerical-contract variants").
* §2.3, Eq. (M-bound): M = ∏ m_i > 2 max|ÃB̃|, symmetric range [-M/2, M/2).
* §2.3, Phase 2, Eq. (modgemm): C^(i) = (Ã mod m_i)(B̃ mod m_i) mod m_i.
* §2.3, Phase 3, Eq. (garner) and Appendix A: Garner mixed-radix digits.
* §2.3 and Algorithm 1: unscale C = D^-1 C̃ E^-1 (exact: powers of two).
* §2.4: the "+1" max-magnitude estimation pass (α = 3r + 1).
* §2.5 "The frozen plane kernel": the published modulus set S, Eq.
  (sq-shortcut), Eq. (kar), the E4M3 envelope Eq. (envelope), the
  carry-corrected base-16 split, and Eq. (accum-exact).
* Algorithm 1 and §2.6 contract item (vi): native-FP64 fallback rows.

Where the paper is silent, this module takes the following readings (the
CUDA path applies the same ones):

R-scale  The "+1" pass computes U = ÂB̂ from power-of-two magnitude planes
         (defined in :func:`magnitude_exponents`); the row/column exponents
         are then chosen so that Σ_l |Ã_il||B̃_lj| ≤ 2^T, where under TZ
         T is the largest integer with 2^(T+1) < M (⌊log2 M⌋ - 1 for the
         products of the moduli used here, none a power of two) and under
         RN two less.  The literal crude bound
         μ = k·max|Ã|·max|B̃| of Algorithm 1 is kept as scale mode "R1".
R-moduli r ≤ 12 takes the prefix of S in the order the paper lists it;
         r = 13..16 appends the primes 479, 467, 463, 461.
R-centre Centred residues lie in [-⌊m/2⌋, m-1-⌊m/2⌋] (= [-m/2, m/2) for
         even m); balanced base-s digits lie in [-⌊s/2⌋, s-1-⌊s/2⌋].
R-fallback A row of A (column of B) takes the native FP64 path when it holds
         a non-finite value, or when its max-exponent lies more than 128
         binades from the lower median over the other nonzero rows
         (columns).  Such rows/columns are treated as zero by the emulated
         path and then overwritten by a sequential FMA chain over l.

Exactness notes.  All integer work uses Python ints or int64.  Two matrix
products use float64 BLAS on integer-valued operands; each call asserts the
bound under which every partial sum is an integer below 2^53, so the product
is exact whatever the summation order.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from fractions import Fraction

import numpy as np

# --------------------------------------------------------------------------
# Moduli (§2.5: the published set S, r = 12, listed as six squares
# 1089, 1024, 961, 841, 625, 529 and the nonsquare tail 511 ... 487).
# --------------------------------------------------------------------------
MODULI_S = (1089, 1024, 961, 841, 625, 529, 511, 509, 503, 499, 491, 487)
# Reading R-moduli: extension primes for r = 13..16 (nonsquare, < 513, so
# inside the carry-corrected envelope of §2.5).
MODULI_EXTENSION = (479, 467, 463, 461)
MAX_MODULI = len(MODULI_S) + len(MODULI_EXTENSION)

E4M3_MAX = 448
NONSQUARE_BASE_BITS = 4          # §2.5: balanced base-16 split, b = 4
NONSQUARE_BASE = 1 << NONSQUARE_BASE_BITS
FALLBACK_EXPONENT_WINDOW = 128   # reading R-fallback


def moduli(r: int) -> tuple:
    """The first r moduli (reading R-moduli)."""
    if not 1 <= r <= MAX_MODULI:
        raise ValueError(f"r must be in [1, {MAX_MODULI}], got {r}")
    return (MODULI_S + MODULI_EXTENSION)[:r]


def square_base(m: int):
    """s with s*s == m, or None for a nonsquare modulus (§2.5)."""
    s = math.isqrt(m)
    return s if s * s == m else None


def modulus_product(mods) -> int:
    """M = ∏ m_i (Eq. M-bound)."""
    M = 1
    for m in mods:
        M *= m
    return M


def range_exponent(mods, quant: str = "tz") -> int:
    """T with 2^T bounding Σ_l |Ã_il||B̃_lj| (reading R-scale).

    TZ: the largest T with 2^T < M/2 (Eq. M-bound), i.e. 2^(T+1) < M.
    RN: two bits less, because rounding to nearest can at most double a
    magnitude (|round(x)| ≤ 2|x| for every real x), so Σ|Ã||B̃| ≤ 4·2^T.
    """
    M = modulus_product(mods)
    t_tz = (M - 1).bit_length() - 2
    return t_tz if quant == "tz" else t_tz - 2


# --------------------------------------------------------------------------
# E4M3 (§2.4: 4 exponent bits, 3 fraction bits, max finite 448; consecutive
# integers exact only on [-16, 16]).  The encoder below is written from the
# format definition: code = sign<<7 | biased_exponent<<3 | fraction, bias 7.
# --------------------------------------------------------------------------
def e4m3_exact_integer(x: int) -> bool:
    """Membership of the set 𝔼 of §2.5: integers M·2^e with |M| ≤ 15, |x| ≤ 448."""
    x = abs(int(x))
    if x == 0:
        return True
    if x > E4M3_MAX:
        return False
    while x % 2 == 0:
        x //= 2
    return x <= 15


def e4m3_encode_integer(x: int) -> int:
    """Byte code of an integer in 𝔼 (raises if the integer is not exact)."""
    x = int(x)
    if not e4m3_exact_integer(x):
        raise ValueError(f"{x} is not exactly representable in E4M3")
    if x == 0:
        return 0
    sign = 0x80 if x < 0 else 0
    a = abs(x)
    e = a.bit_length() - 1               # a = 1.fff × 2^e, e ≥ 0
    frac_times_8 = (a << 3) // (1 << e) - 8
    assert (a << 3) % (1 << e) == 0 and 0 <= frac_times_8 < 8
    return sign | ((e + 7) << 3) | frac_times_8


def e4m3_encode_power_of_two(q: int) -> int:
    """Byte code of 2^q for q in [-9, 8] (normal for q ≥ -6, else subnormal)."""
    if not -9 <= q <= 8:
        raise ValueError("2^q is outside the E4M3 range")
    if q >= -6:
        return (q + 7) << 3
    return 1 << (q + 9)                  # subnormal: f/8 · 2^-6 with f = 2^(q+9)


def e4m3_decode(code: int) -> float:
    """Value of an E4M3 byte, written from the format definition."""
    sign = -1.0 if code & 0x80 else 1.0
    e = (code >> 3) & 0xF
    f = code & 0x7
    if e == 0xF and f == 0x7:
        return math.nan
    if e == 0:
        return sign * (f / 8.0) * 2.0 ** -6
    return sign * (1.0 + f / 8.0) * 2.0 ** (e - 7)


_ENCODE_TABLE = {v: e4m3_encode_integer(v) for v in range(-E4M3_MAX, E4M3_MAX + 1)
                 if e4m3_exact_integer(v)}


def e4m3_encode_array(x: np.ndarray) -> np.ndarray:
    """Vectorised :func:`e4m3_encode_integer` over an integer array."""
    x = np.asarray(x, dtype=np.int64)
    out = np.empty(x.shape, dtype=np.uint8)
    flat_in, flat_out = x.ravel(), out.ravel()
    for v in np.unique(flat_in):
        flat_out[flat_in == v] = _ENCODE_TABLE[int(v)]
    return out


# --------------------------------------------------------------------------
# Centred residues and the digit-plane layout (§2.5).
# --------------------------------------------------------------------------
def centred(x, m: int):
    """Representative of x mod m in [-⌊m/2⌋, m-1-⌊m/2⌋] (reading R-centre)."""
    x = np.asarray(x, dtype=np.int64)
    r = np.mod(x, m)
    return np.where(r > m - 1 - m // 2, r - m, r)


def square_digits(d, s: int):
    """Balanced base-s digits of a centred residue: d = d0 + s·d1 (Eq. sq-shortcut)."""
    d = np.asarray(d, dtype=np.int64)
    h = s // 2
    d0 = np.mod(d + h, s) - h
    d1 = (d - d0) // s
    return d0, d1


def nonsquare_digits(d):
    """Carry-corrected balanced base-16 digits, d = d0 + 16·d1 (§2.5).

    Start from the balanced base-16 digits d0 ∈ [-8, 7]; when d0 + d1 is not in
    𝔼, move one unit of base weight: (d0, d1) ↦ (d0 - 16ς, d1 + ς), ς = sign d0.
    """
    d = np.asarray(d, dtype=np.int64)
    B = NONSQUARE_BASE
    d0 = np.mod(d + B // 2, B) - B // 2
    d1 = (d - d0) // B
    in_e = np.vectorize(e4m3_exact_integer, otypes=[bool])(d0 + d1) if d.size else np.zeros(0, bool)
    sig = np.sign(d0)
    d0c = np.where(in_e, d0, d0 - B * sig)
    d1c = np.where(in_e, d1, d1 + sig)
    return d0c, d1c


def digit_planes(d, m: int, merged: bool = False):
    """Integer planes stored for one operand and one modulus (§2.5).

    Square m = s²: (d0, d1).  Nonsquare: (d0 + d1, d0, d1) -- the sum plane
    first, as the Karatsuba product pairs sum with sum.  With ``merged`` the
    last plane is stored pre-scaled by -2^b (the accumulator merge of §2.5,
    "Accumulators"); only the A operand uses the pre-scaled plane.
    """
    s = square_base(m)
    if s is not None:
        d0, d1 = square_digits(d, s)
        return [d0, d1]
    d0, d1 = nonsquare_digits(d)
    last = -NONSQUARE_BASE * d1 if merged else d1
    return [d0 + d1, d0, last]


def plane_product_value(pa, pb, m: int, merged: bool = False):
    """Recombine per-element plane products into d·e (mod m), §2.5.

    Square, Eq. (sq-shortcut): d0e0 + s(d1e0 + d0e1) ≡ de (mod s²).
    Nonsquare, Eq. (kar) with b = 4:
        de = (1-2^b) d0e0 + 2^b (d0+d1)(e0+e1) + (2^2b - 2^b) d1e1.
    Merged: acc = d0e0 - 2^b d1e1 carries the common weight (1 - 2^b).
    ``pa``/``pb`` are plane lists from :func:`digit_planes` (A merged, B not).
    """
    s = square_base(m)
    if s is not None:
        a0, a1 = pa
        b0, b1 = pb
        return a0 * b0 + s * (a1 * b0 + a0 * b1)
    B = NONSQUARE_BASE
    asum, a0, a1 = pa
    bsum, b0, b1 = pb
    if merged:
        return B * (asum * bsum) + (1 - B) * (a0 * b0 + a1 * b1)
    return B * (asum * bsum) + (1 - B) * (a0 * b0) + (B * B - B) * (a1 * b1)


def plane_counts(mods):
    """(p_store, p_mma, N_acc) of §2.5 "Three distinct counts" (unmerged tail)."""
    p_store = sum(2 if square_base(m) else 3 for m in mods)
    p_mma = 3 * len(mods)
    n_acc = sum(2 if square_base(m) else 3 for m in mods)
    return p_store, p_mma, n_acc


# --------------------------------------------------------------------------
# Exponents (§2.3 Phase 1; Algorithm 1 "scan the exponent spans"; App. C).
# --------------------------------------------------------------------------
def frexp_exponent(x):
    """e with x = f·2^e, 0.5 ≤ |f| < 1 (0 for x = 0); so |x| < 2^e."""
    _, e = np.frexp(np.asarray(x, dtype=np.float64))
    return e.astype(np.int64)


def ceil_log2_abs(x):
    """⌈log2 |x|⌉ for finite nonzero doubles, exactly, from the binary exponent."""
    f, e = np.frexp(np.abs(np.asarray(x, dtype=np.float64)))
    e = e.astype(np.int64)
    return np.where(f == 0.5, e - 1, e)


def ceil_log2_int(x):
    """⌈log2 x⌉ for positive integers below 2^53."""
    return ceil_log2_abs(np.asarray(x, dtype=np.float64))


def fallback_flags(exps, nonfinite, nonzero):
    """Reading R-fallback for one operand's rows (A) or columns (B).

    Flag a row holding a non-finite value, or one whose max-exponent lies more
    than 128 binades from the lower median of the exponents of the nonzero,
    finite rows.  Returns (flags, median).
    """
    exps = np.asarray(exps, dtype=np.int64)
    cand = nonzero & ~nonfinite
    flags = nonfinite.copy()
    med = 0
    if cand.any():
        srt = np.sort(exps[cand])
        med = int(srt[(srt.size - 1) // 2])
        flags |= cand & (np.abs(exps - med) > FALLBACK_EXPONENT_WINDOW)
    return flags, med


def scan_rows(X):
    """Per row of X (rows × k): max-exponent, non-finite flag, nonzero flag.

    The max-exponent is the frexp exponent of the largest finite magnitude, so
    every |X_il| < 2^e_i (Algorithm 1 "scan the exponent spans"; App. C).
    """
    X = np.asarray(X, dtype=np.float64)
    finite = np.isfinite(X)
    nonfinite = ~finite.all(axis=1) if X.shape[1] else np.zeros(X.shape[0], bool)
    mag = np.where(finite, np.abs(X), 0.0)
    mx = mag.max(axis=1) if X.shape[1] else np.zeros(X.shape[0])
    return frexp_exponent(mx), nonfinite, mx > 0


def magnitude_clamp(k: int) -> int:
    """c = ⌊(24 - ⌈log2 k⌉)/2⌋ clamped to [0, 9] (reading R-scale).

    It makes every product of two magnitude-plane entries a multiple of 2^-2c
    and keeps U·2^2c ≤ k·2^2c ≤ 2^24, so the FP32 "+1" GEMM is exact; 9 is the
    smallest E4M3 exponent (2^-9, subnormal).
    """
    lk = 0 if k <= 1 else int(k - 1).bit_length()
    return max(0, min(9, (24 - lk) // 2))


def magnitude_exponents(X, e_rows, c: int, zero_rows=None):
    """Exponent q_il of the magnitude plane X̂_il = 2^q_il (0 entries → None).

    q = max(-c, ⌈log2(|X_il| · 2^-e_i)⌉), computed as ⌈log2|X_il|⌉ - e_i on
    integers, so X̂_il ≥ |X_il|·2^-e_i and X̂_il ∈ [2^-c, 1].  Returns an
    int64 array with -10**6 marking zero entries (and rows in ``zero_rows``).
    """
    X = np.asarray(X, dtype=np.float64)
    nz = (X != 0) & np.isfinite(X)
    if zero_rows is not None:
        nz &= ~zero_rows[:, None]
    q = np.full(X.shape, -10**6, dtype=np.int64)
    cl = ceil_log2_abs(np.where(nz, X, 1.0)) - e_rows[:, None]
    q[nz] = np.maximum(-c, cl[nz])
    return q


def exact_int_matmul(a, b, bound_a: int, bound_b: int):
    """Exact product of integer matrices through float64 BLAS.

    Exact because every product and every partial sum is an integer of
    magnitude ≤ k·bound_a·bound_b < 2^53 (asserted), which float64 holds.
    """
    k = a.shape[1]
    assert k * bound_a * bound_b < 2**53, "exactness bound of the float64 product"
    assert np.abs(a).max(initial=0) <= bound_a and np.abs(b).max(initial=0) <= bound_b
    return (a.astype(np.float64) @ b.astype(np.float64)).astype(np.int64)


def plus_one_pass(qa, qb, c: int):
    """The "+1" max-magnitude estimation GEMM (§2.4) on power-of-two planes.

    Returns U·2^2c as exact int64 (Â·2^c and B̂·2^c are integers in [1, 2^c]).
    ``qa`` is rows(A) × k, ``qb`` is k × cols(B).
    """
    ia = np.where(qa > -10**5, np.left_shift(1, np.maximum(qa + c, 0)), 0).astype(np.int64)
    ib = np.where(qb > -10**5, np.left_shift(1, np.maximum(qb + c, 0)), 0).astype(np.int64)
    return exact_int_matmul(ia, ib, 1 << c, 1 << c)


def choose_scales(U2c, c: int, ra, cb, T: int, zero_rows, zero_cols):
    """Row exponents d_i and column exponents e_j (reading R-scale, mode R2).

    u_i = max_j ⌈log2 U_ij⌉ (rows without a positive entry take u_max; u_max
    = 0 when U vanishes), s = min(62, ⌊(T - u_max)/2⌋), t_i = min(62, T - s - u_i),
    d_i = t_i - ra_i, e_j = s - cb_j.  Since |A_il| 2^-ra_i ≤ Â_il, TZ gives
    |Ã_il| ≤ 2^t_i Â_il and |B̃_lj| ≤ 2^s B̂_lj, hence
        Σ_l |Ã_il||B̃_lj| ≤ 2^(t_i+s) U_ij ≤ 2^T < M/2   (Eq. M-bound).
    """
    m, n = U2c.shape
    pos = U2c > 0
    u = np.full(m, np.iinfo(np.int64).min, dtype=np.int64)
    if n:
        cl = np.where(pos, ceil_log2_int(np.where(pos, U2c, 1)) - 2 * c, np.iinfo(np.int64).min)
        u = cl.max(axis=1)
    has = pos.any(axis=1) if n else np.zeros(m, bool)
    u_max = int(u[has].max()) if has.any() else 0
    u = np.where(has, u, u_max)
    s = min(62, (T - u_max) // 2)
    t = np.minimum(62, T - s - u)
    d = t - ra
    e = s - cb
    d = np.where(zero_rows, 0, d)
    e = np.where(zero_cols, 0, e)
    return d.astype(np.int64), e.astype(np.int64), u, u_max, s


def choose_scales_r1(k: int, ra, cb, T: int, zero_rows, zero_cols):
    """Scale mode R1: the literal bound μ = k·max|Ã|·max|B̃| of Algorithm 1.

    |Ã_il| < 2^pA and |B̃_lj| < 2^pB with pA + pB + ⌈log2 k⌉ = T.
    """
    lk = 0 if k <= 1 else int(k - 1).bit_length()
    pA = min(62, (T - lk) // 2)
    pB = min(62, T - lk - pA)
    d = np.where(zero_rows, 0, pA - ra)
    e = np.where(zero_cols, 0, pB - cb)
    return d.astype(np.int64), e.astype(np.int64)


def quantise(X, exps_rows, quant: str = "tz"):
    """Ã = ⌊D X⌉ with D = diag(2^d_i) (Eq. scale; Table "numerical-contract variants").

    ldexp by a power of two is exact whenever the result is ≥ 1/2 in
    magnitude, and smaller results quantise to 0 under both rules.
    """
    X = np.asarray(X, dtype=np.float64)
    Y = np.ldexp(np.where(np.isfinite(X), X, 0.0), exps_rows[:, None])
    if quant == "tz":
        Q = np.trunc(Y)
    elif quant == "rn":
        Q = np.rint(Y)                  # round half to even
    else:
        raise ValueError(quant)
    assert np.all(np.abs(Q) <= 2.0**62)
    return Q.astype(np.int64)


# --------------------------------------------------------------------------
# Phase 2 (Eq. modgemm) and Phase 3 (Eq. garner, Appendix A).
# --------------------------------------------------------------------------
def residue_products(At, Bt, mods):
    """C^(i) = centred((Ã mod m_i)(B̃ mod m_i) mod m_i) for each modulus."""
    out = []
    for m in mods:
        a = centred(At, m)
        b = centred(Bt, m)
        h = m - m // 2
        out.append(centred(exact_int_matmul(a, b, h, h), m))
    return np.stack(out) if out else np.zeros((0,) + (At.shape[0], Bt.shape[1]), np.int64)


def garner_digits(res, mods):
    """Mixed-radix digits v_k ∈ [0, m_k) of Eq. (garner).

    v_1 = C^(1) mod m_1;  v_k = (C^(k) - Σ_{j<k} v_j P_{j-1}) · P_{k-1}^{-1} mod m_k
    with P_j = m_1 ⋯ m_j (P_0 = 1).  ``res`` has shape (r, ...).
    """
    res = np.asarray(res, dtype=np.int64)
    v = []
    for k, mk in enumerate(mods):
        acc = res[k] % mk
        P = 1
        for j in range(k):
            acc = (acc - v[j] * (P % mk)) % mk
            P *= mods[j]
        inv = pow(P % mk, -1, mk) if k else 1
        v.append((acc * inv) % mk)
    return v


def garner_value(res, mods):
    """X = Σ_k v_k P_{k-1} mapped to [-M/2, M/2) (Eq. M-bound), as Python ints."""
    v = garner_digits(res, mods)
    M = modulus_product(mods)
    shape = np.asarray(res).shape[1:]
    X = np.zeros(shape, dtype=object)
    P = 1
    for k, mk in enumerate(mods):
        X = X + v[k].astype(object) * P
        P *= mk
    return np.where(2 * X >= M, X - M, X)


def unscale_one(X: int, E: int) -> float:
    """Correctly rounded (RNE) float64 of X · 2^E (§2.3 Phase 3: C = D^-1 C̃ E^-1).

    float(int) rounds once; scaling by 2^E is then exact unless the result is
    subnormal, in which case the exact rational is rounded once instead.
    """
    X = int(X)
    if X == 0:
        return 0.0
    top = X.bit_length() if X > 0 else (-X).bit_length()
    if top - 1 + E >= -1022:                       # normal (or overflow)
        try:
            return math.ldexp(float(X), E)
        except OverflowError:
            return math.copysign(math.inf, X)
    return float(Fraction(X) * Fraction(2) ** E)


def unscale(X, d, e):
    m, n = X.shape
    C = np.empty((m, n), dtype=np.float64)
    for i in range(m):
        for j in range(n):
            C[i, j] = unscale_one(X[i, j], -int(d[i]) - int(e[j]))
    return C


# --------------------------------------------------------------------------
# Native-FP64 fallback (Algorithm 1, the "if" on admissibility; §2.6 (vi)).
# --------------------------------------------------------------------------
def fma(a: float, b: float, c: float) -> float:
    """Correctly rounded a·b + c (IEEE 754 fusedMultiplyAdd, RNE)."""
    if math.isfinite(a) and math.isfinite(b):
        if not math.isfinite(c):
            return c
        exact = Fraction(a) * Fraction(b) + Fraction(c)
        if exact == 0:
            # An exact zero is -0 only when the product and c are both -0.
            if (a == 0 or b == 0) and c == 0:
                neg_p = math.copysign(1.0, a) * math.copysign(1.0, b) < 0
                if neg_p and math.copysign(1.0, c) < 0:
                    return -0.0
            return 0.0
        try:
            return float(exact)
        except OverflowError:
            return math.copysign(math.inf, exact)
    return a * b + c


def native_entry(A, B, i: int, j: int) -> float:
    """C_ij = FMA chain over l = 0..k-1 starting from +0.0."""
    s = 0.0
    for l in range(A.shape[1]):
        s = fma(float(A[i, l]), float(B[l, j]), s)
    return s


# --------------------------------------------------------------------------
# Algorithm 1 end to end.
# --------------------------------------------------------------------------
@dataclass
class Result:
    C: np.ndarray
    mods: tuple
    T: int
    c: int
    ra: np.ndarray
    cb: np.ndarray
    row_flag: np.ndarray
    col_flag: np.ndarray
    qa: np.ndarray = None
    qb: np.ndarray = None
    U2c: np.ndarray = None
    u: np.ndarray = None
    u_max: int = 0
    s: int = 0
    d: np.ndarray = None
    e: np.ndarray = None
    At: np.ndarray = None
    Bt: np.ndarray = None
    residues: np.ndarray = None
    X: np.ndarray = None
    extra: dict = field(default_factory=dict)


def prepare(A, B, r: int = 12, quant: str = "tz", scale: str = "r2", fallback: bool = True) -> Result:
    """Phase 1 of Algorithm 1 and the scale choice, on the whole problem.

    Returns a Result without C: exponents, flags, the "+1" pass, d, e, the
    integer matrices Ã, B̃ (Eq. scale) and the centred residues of B̃ for each
    modulus (Algorithm 1 "lin:dec" for B, needed by every row of C).
    """
    A = np.asarray(A, dtype=np.float64)
    B = np.asarray(B, dtype=np.float64)
    m, k = A.shape
    k2, n = B.shape
    assert k == k2
    mods = moduli(r)
    T = range_exponent(mods, quant)
    c = magnitude_clamp(k)

    # Phase 1 scan: exponents, non-finite rows/columns, fallback flags.
    ra, nfa, nza = scan_rows(A)
    cb, nfb, nzb = scan_rows(B.T)
    if fallback:
        row_flag, _ = fallback_flags(ra, nfa, nza)
        col_flag, _ = fallback_flags(cb, nfb, nzb)
    else:
        row_flag, col_flag = nfa.copy(), nfb.copy()
    zero_rows = row_flag | ~nza          # rows the emulated path treats as 0
    zero_cols = col_flag | ~nzb
    ra = np.where(zero_rows, 0, ra)
    cb = np.where(zero_cols, 0, cb)

    res = Result(C=None, mods=mods, T=T, c=c, ra=ra, cb=cb,
                 row_flag=row_flag, col_flag=col_flag)

    # "+1" pass and the choice of D, E.
    if scale == "r2":
        qa = magnitude_exponents(A, ra, c, zero_rows)
        qb = magnitude_exponents(B.T, cb, c, zero_cols)
        U2c = plus_one_pass(qa, qb.T, c)
        d, e, u, u_max, s = choose_scales(U2c, c, ra, cb, T, zero_rows, zero_cols)
        res.qa, res.qb, res.U2c, res.u, res.u_max, res.s = qa, qb, U2c, u, u_max, s
    elif scale == "r1":
        d, e = choose_scales_r1(k, ra, cb, T, zero_rows, zero_cols)
    else:
        raise ValueError(scale)
    res.d, res.e = d, e

    # Eq. (scale): integer matrices (flagged rows/columns are zero here).
    res.At = quantise(np.where(zero_rows[:, None], 0.0, A), d, quant)
    res.Bt = quantise(np.where(zero_cols[:, None], 0.0, B.T), e, quant).T
    # Centred residues of B̃, held as float64 (exact: |residue| ≤ 544) with
    # the bound of exact_int_matmul checked once here.
    bres = []
    for mi in mods:
        b = centred(res.Bt, mi)
        h = mi - mi // 2
        assert np.abs(b).max(initial=0) <= h and k * h * h < 2**53
        bres.append(b.astype(np.float64))
    res.extra["b_residues"] = bres
    return res


def evaluate_rows(prep: Result, A, B, rows=None) -> Result:
    """Phases 2-3 (Eq. modgemm, Eq. garner, unscale) and the native fallback
    for the given rows of C (all rows when ``rows`` is None)."""
    A = np.asarray(A, dtype=np.float64)
    B = np.asarray(B, dtype=np.float64)
    m, n = A.shape[0], B.shape[1]
    mods = prep.mods
    sel = np.arange(m) if rows is None else np.asarray(rows, dtype=np.int64)
    At = prep.At[sel]
    out = []
    for mi, b in zip(mods, prep.extra["b_residues"]):
        # exact: every partial sum is an integer below k·(m/2)^2 < 2^53
        a = centred(At, mi).astype(np.float64)
        out.append(centred((a @ b).astype(np.int64), mi))
    R = np.stack(out) if out else np.zeros((0, sel.size, n), np.int64)
    X = garner_value(R, mods)
    C = unscale(X, prep.d[sel], prep.e)
    # Native FP64 on flagged rows and columns.
    for a, i in enumerate(sel):
        if prep.row_flag[i]:
            for j in range(n):
                C[a, j] = native_entry(A, B, i, j)
    for j in np.flatnonzero(prep.col_flag):
        for a, i in enumerate(sel):
            if not prep.row_flag[i]:
                C[a, j] = native_entry(A, B, i, j)
    res = Result(**{f: getattr(prep, f) for f in prep.__dataclass_fields__})
    res.residues, res.X, res.C = R, X, C
    return res


def oz2_dgemm(A, B, r: int = 12, quant: str = "tz", scale: str = "r2",
              fallback: bool = True, rows=None) -> Result:
    """C ≈ AB by Ozaki Scheme II (Algorithm 1), every intermediate returned.

    With ``rows`` (an index array) Phase 1 and the scale choice still run on
    the whole problem, but Phases 2-3 and the fallback are evaluated only for
    those rows of C (``C``, ``residues`` and ``X`` then hold those rows).
    """
    return evaluate_rows(prepare(A, B, r, quant, scale, fallback), A, B, rows)


def truncation_bound(A, B, d, e, quant: str = "tz"):
    """Per-entry bound on |C - AB| from the quantiser alone (App. C).

    TZ: |X 2^d - ⌊X 2^d⌋| < 1, so |A_il - Ã_il 2^-d_i| < 2^-d_i, and
        |C - AB|_ij ≤ Σ_l (2^-d_i |B_lj| + |A_il| 2^-e_j + 2^-d_i-e_j) + u|C_ij|.
    RN halves each quantisation term.
    """
    A = np.asarray(A, dtype=np.float64)
    B = np.asarray(B, dtype=np.float64)
    h = 1.0 if quant == "tz" else 0.5
    sa = np.ldexp(h, -d)[:, None]
    sb = np.ldexp(h, -e)[None, :]
    absA, absB = np.abs(A), np.abs(B)
    k = A.shape[1]
    return sa * absB.sum(axis=0)[None, :] + absA.sum(axis=1)[:, None] * sb + k * sa * sb
