// Device arithmetic of Phase 3 (§2.3 Eq. garner, Appendix A; Algorithm 1
// "C ← D^-1 C̃ E^-1"), shared by the reconstruction kernel and the fused
// residue-GEMM + reconstruction kernel: from the residues c_k of an output,
// the integer X ∈ [-M/2, M/2) and one correctly rounded conversion of
// X·2^E to FP64.  Garner's algorithm (crt_value) defines the result; the
// direct-CRT forms reach the same value with multiply-adds only.
#pragma once

#include "oz2_common.cuh"

namespace oz2 {

typedef unsigned long long u64;
typedef unsigned __int128 u128;


// X (L little-endian 32-bit limbs) = X·m + v.  Only the low `nl` limbs can be
// nonzero afterwards; each limb step is one 32×32+64-bit multiply-add.
template <int L>
__device__ __forceinline__ void horner_step(uint32_t (&w)[L], int nl, uint32_t m, uint32_t v) {
  u64 t = static_cast<u64>(w[0]) * m + v;
  w[0] = static_cast<uint32_t>(t);
#pragma unroll
  for (int i = 1; i < L; ++i) {
    if (i < nl) {
      t = static_cast<u64>(w[i]) * m + (t >> 32);
      w[i] = static_cast<uint32_t>(t);
    }
  }
}

// Nearest double (ties to even) to (-1)^neg · (x + δ) · 2^E, where δ ∈ [0, 1)
// is nonzero exactly when `sticky` is set (bits already shifted out of x).
__device__ __forceinline__ double round_to_double(u64 x, bool sticky, int E, bool neg) {
  const u64 sign = neg ? (1ull << 63) : 0ull;
  if (x == 0) return __longlong_as_double(static_cast<long long>(sign));
  const int Lb = 64 - __clzll(static_cast<long long>(x));
  const int top = Lb - 1 + E;  // exponent of the leading bit
  if (top > 1023) return __longlong_as_double(static_cast<long long>(sign | 0x7FF0000000000000ull));
  const int p = top >= -1022 ? 53 : top + 1075;  // significant bits available
  const int sh = Lb - p;                         // bits to drop (≤ 63)
  u64 q;
  if (sh <= 0) {
    q = x << (-sh);  // Lb ≤ p ≤ 53; no bits were shifted out (sticky implies Lb = 64)
  } else if (p <= 0) {
    // Below the smallest subnormal: round up only when strictly above half of it.
    const bool below = (x & ((1ull << (Lb - 1)) - 1)) != 0 || sticky;
    q = (p == 0 && below) ? 1 : 0;
  } else {
    q = x >> sh;
    const bool rbit = ((x >> (sh - 1)) & 1) != 0;
    const bool st = sticky || (x & ((1ull << (sh - 1)) - 1)) != 0;
    if (rbit && (st || (q & 1))) ++q;
  }
  if (q == 0) return __longlong_as_double(static_cast<long long>(sign));
  if (p < 53) return __longlong_as_double(static_cast<long long>(sign | q));  // q · 2^-1074 (2^52: smallest normal)
  int f = top;  // q ∈ [2^52, 2^53]
  if (q >> 53) {
    q >>= 1;
    ++f;
  }
  if (f > 1023) return __longlong_as_double(static_cast<long long>(sign | 0x7FF0000000000000ull));
  return __longlong_as_double(
      static_cast<long long>(sign | (static_cast<u64>(f + 1023) << 52) | (q & ((1ull << 52) - 1))));
}

// (a·w) mod m for a < 2^32 and a fixed w < m with wp = ⌊w·2^32/m⌋ (V. Shoup's
// modular multiplication with a precomputed quotient): q = ⌊a·wp/2^32⌋ is
// the true quotient or one less, so a·w - q·m ∈ [0, 2m).
__device__ __forceinline__ uint32_t mulmod_shoup(uint32_t a, uint32_t w, uint32_t wp, uint32_t m) {
  const uint32_t q = __umulhi(a, wp);
  const uint32_t r = a * w - q * m;
  return r >= m ? r - m : r;
}

// One output: centred residues c[0..R) → nearest double of X·2^E.
template <int R>
__device__ __forceinline__ double crt_value(const int (&c)[R], int E, const Oz2Moduli& mods) {
  // Garner digits (Eq. garner): v_k = (c_k - Σ_{j<k} v_j P_{j-1}) P_{k-1}^{-1} mod m_k,
  // with (P_{j-1} mod m_k) precomputed.  The sums are carried for every later
  // modulus as soon as a digit is known, so each digit waits on one
  // multiply-add; goff_k (a multiple of m_k ≥ 2^27) keeps them positive.
  int S[R];
#pragma unroll
  for (int k = 0; k < R; ++k) S[k] = mods.goff[k] + c[k];
  uint32_t v[R];
#pragma unroll
  for (int k = 0; k < R; ++k) {
    v[k] = mulmod_shoup(static_cast<uint32_t>(S[k]), static_cast<uint32_t>(mods.inv[k]), mods.invp[k],
                        static_cast<uint32_t>(mods.m[k]));
#pragma unroll
    for (int j = k + 1; j < R; ++j) S[j] -= static_cast<int>(v[k]) * mods.pmod[j][k];
  }
  // Mixed radix → integer by Horner from the top digit; after j steps the value
  // is below the product of j+1 moduli < 2^(11(j+1)), which bounds the limbs.
  constexpr int L = R <= 12 ? 4 : 5;  // M < 2^112 (r ≤ 12), < 2^148 (r ≤ 16)
  uint32_t w[L];
  w[0] = v[R - 1];
#pragma unroll
  for (int i = 1; i < L; ++i) w[i] = 0;
#pragma unroll
  for (int k = R - 2; k >= 0; --k) {
    const int nl = (11 * (R - k) + 31) / 32 < L ? (11 * (R - k) + 31) / 32 : L;
    horner_step<L>(w, nl, static_cast<uint32_t>(mods.m[k]), v[k]);
  }
  // Symmetric range [-M/2, M/2) (Eq. M-bound): X ≥ ⌈M/2⌉ ⇔ 2X ≥ M.
  bool ge = true, decided = false;
#pragma unroll
  for (int i = L - 1; i >= 0; --i) {
    const uint32_t h = static_cast<uint32_t>(mods.Mhalf[i >> 1] >> (32 * (i & 1)));
    if (!decided && w[i] != h) {
      ge = w[i] > h;
      decided = true;
    }
  }
  const bool neg = ge;
  if (neg) {  // |X - M| = M - X
    uint32_t borrow = 0;
#pragma unroll
    for (int i = 0; i < L; ++i) {
      const u64 t = static_cast<u64>(static_cast<uint32_t>(mods.M[i >> 1] >> (32 * (i & 1)))) - w[i] - borrow;
      w[i] = static_cast<uint32_t>(t);
      borrow = static_cast<uint32_t>(t >> 63);
    }
  }
  // Leading 64 bits and a sticky bit for everything below them.
  u128 x = (static_cast<u128>(w[3]) << 96) | (static_cast<u128>(w[2]) << 64) | (static_cast<u128>(w[1]) << 32) | w[0];
  bool sticky = false;
  if (L == 5 && w[L - 1] != 0) {
    sticky = w[0] != 0;
    x = (static_cast<u128>(w[L - 1]) << 96) | (x >> 32);
    E += 32;
  }
  const u64 xh = static_cast<u64>(x >> 64);
  u64 top64 = static_cast<u64>(x);
  if (xh) {
    const int s = 64 - __clzll(static_cast<long long>(xh));  // bits above the low word
    top64 = (xh << (64 - s)) | (static_cast<u64>(x) >> s);
    sticky = sticky || (static_cast<u64>(x) << (64 - s)) != 0;
    E += s;
  }
  return round_to_double(top64, sticky, E, neg);
}

// The five-limb direct CRT (any r ≤ 16; the exact path tries it before
// Garner for r ≥ 13): the same X by the direct CRT sum, kept exact over
// six 32-bit limbs.  With u_k = c_k + coff_k ≥ 0,
// S = Σ_k u_k W_k ≡ X (mod M), and S/M = Σ_k u_k y_k/m_k, so
// q = ⌊S/M + 1/2⌋ gives X = S - q·M ∈ [-M/2, M/2).  q comes from the
// 32.32 fixed-point sum Σ u_k F_k + 2^31, whose error is below
// Σ u_k·2^-33 < 2^-13.3; when its fraction is within 2^19/2^32 of an integer
// (X within that margin of ±M/2, which products bounded by Eq. M-bound never
// reach) the caller falls back to Garner.  Returns false in that case.
template <int R>
__device__ __forceinline__ bool crt_value_fast(const int (&c)[R], int E, const Oz2Moduli& mods, double& out) {
  constexpr int LW = R <= 12 ? 4 : 5;  // limbs of W_k (< M)
  constexpr int LS = LW + 1;           // limbs of S (u_k < 2^16.1, r ≤ 16)
  u64 acc[LS];
#pragma unroll
  for (int j = 0; j < LS; ++j) acc[j] = 0;
  u64 Q = 1ull << 31;
#pragma unroll
  for (int k = 0; k < R; ++k) {
    const uint32_t u = static_cast<uint32_t>(c[k] + mods.coff[k]);
#pragma unroll
    for (int j = 0; j < LW; ++j) acc[j] += static_cast<u64>(u) * mods.crtw[k][j];
    Q += static_cast<u64>(u) * mods.crtf[k];
  }
  const uint32_t frac = static_cast<uint32_t>(Q);
  if (frac < (1u << 19) || frac > 0xFFFFFFFFu - (1u << 19)) return false;
  const uint32_t q = static_cast<uint32_t>(Q >> 32);
  // x = S - q·M, two's complement over LS limbs.
  uint32_t x[LS];
  u64 sc = 0, pc = 0;
  uint32_t borrow = 0;
#pragma unroll
  for (int j = 0; j < LS; ++j) {
    const u64 sj = acc[j] + sc;
    sc = sj >> 32;
    const uint32_t mj = j < 6 ? static_cast<uint32_t>(mods.M[j >> 1] >> (32 * (j & 1))) : 0u;
    const u64 pj = static_cast<u64>(q) * mj + pc;
    pc = pj >> 32;
    const u64 dj = static_cast<u64>(static_cast<uint32_t>(sj)) - static_cast<uint32_t>(pj) - borrow;
    x[j] = static_cast<uint32_t>(dj);
    borrow = static_cast<uint32_t>(dj >> 63);
  }
  const bool neg = (x[LS - 1] >> 31) != 0;
  if (neg) {  // magnitude of the two's complement value
    uint32_t cy = 1;
#pragma unroll
    for (int j = 0; j < LS; ++j) {
      const u64 t = static_cast<u64>(~x[j]) + cy;
      x[j] = static_cast<uint32_t>(t);
      cy = static_cast<uint32_t>(t >> 32);
    }
  }
  // |X| < M/2 fits in LW limbs; leading 64 bits and a sticky bit.
  u128 v = (static_cast<u128>(x[3]) << 96) | (static_cast<u128>(x[2]) << 64) | (static_cast<u128>(x[1]) << 32) | x[0];
  bool sticky = false;
  if (LW == 5 && x[LW - 1] != 0) {
    sticky = x[0] != 0;
    v = (static_cast<u128>(x[LW - 1]) << 96) | (v >> 32);
    E += 32;
  }
  const u64 vh = static_cast<u64>(v >> 64);
  u64 top64 = static_cast<u64>(v);
  if (vh) {
    const int s = 64 - __clzll(static_cast<long long>(vh));
    top64 = (vh << (64 - s)) | (static_cast<u64>(v) >> s);
    sticky = sticky || (static_cast<u64>(v) << (64 - s)) != 0;
    E += s;
  }
  out = round_to_double(top64, sticky, E, neg);
  return true;
}

// c·(hi·2^32 + lo) mod 2^64 split as a 64-bit part and a 32-bit high-word
// part: one signed 32×32→64 multiply-add and one 32-bit multiply-add.
__device__ __forceinline__ void mad_word(int c, int lo, int hi, long long& acc64, uint32_t& acc_hi) {
  acc64 += static_cast<long long>(c) * lo;
  acc_hi += static_cast<uint32_t>(c) * static_cast<uint32_t>(hi);
}

// Nearest double to (-1)^neg·(hi·2^64 + lo)·2^E for hi ≠ 0 (general path).
__device__ __forceinline__ double round_to_double_big(u64 hi, u64 lo, int E, bool neg) {
  const int sh = 64 - __clzll(static_cast<long long>(hi));
  const u64 top = (hi << (64 - sh)) | (lo >> sh);
  return round_to_double(top, (lo << (64 - sh)) != 0, E + sh, neg);
}

// Nearest double to X·2^E for X = Hs·2^64 + L (two's complement, |X| < 2^127).
// The common case (|X| ≥ 2^64, normal result) takes the leading 64 bits with
// two funnel shifts and lets the hardware conversion round them: a sticky
// bit for the rest is folded into bit 0, below the rounding position (bit
// 10), so the conversion's round-to-nearest-even decides as the exact value
// would.  The exponent is then added to the double's bit pattern.
__device__ __forceinline__ double finish_words(long long Hs, u64 L, int E) {
  const bool neg = Hs < 0;
  u64 hi = static_cast<u64>(Hs), lo = L;
  if (neg) {
    lo = 0ull - L;
    hi = ~hi + (L == 0 ? 1ull : 0ull);
  }
  if (hi == 0) return round_to_double(lo, false, E, neg);
  const uint32_t w3 = static_cast<uint32_t>(hi >> 32), w2 = static_cast<uint32_t>(hi);
  const uint32_t w1 = static_cast<uint32_t>(lo >> 32), w0 = static_cast<uint32_t>(lo);
  const int s = w3 ? __clz(w3) : 32 + __clz(w2);  // leading zeros of hi (8..63 for |X| < 2^120)
  const int e2 = E + 127 - s;                      // exponent of the leading bit of X·2^E
  if (e2 < -1022 || e2 > 1022) return round_to_double_big(hi, lo, E, neg);
  const bool ge = s >= 32;
  const uint32_t x3 = ge ? w2 : w3, x2 = ge ? w1 : w2, x1 = ge ? w0 : w1, x0 = ge ? 0u : w0;
  const int sp = s & 31;
  const uint32_t th = __funnelshift_l(x2, x3, sp), tl = __funnelshift_l(x1, x2, sp);
  const bool sticky = ((x1 << sp) | x0) != 0;
  const u64 top = (static_cast<u64>(th) << 32) | tl | (sticky ? 1ull : 0ull);  // bit 63 set
  const long long bits = __double_as_longlong(__ull2double_rn(top)) + (static_cast<long long>(E + 64 - s) << 52);
  return __longlong_as_double(bits | (neg ? (1ll << 63) : 0ll));
}

// Fast path for r ≤ 12 (M < 2^112) in 32- and 64-bit words.  With
// S = Σ_k c_k W_k (≡ X mod M) and W_k/M = y_k/m_k:
//  * Y = Σ c_k F_k mod 2^64, read as a signed word, is 2^64·X/M up to
//    Σ|c_k|/2 units, as long as X/M is not within that of ±1/2;
//  * q = (S - X)/M is the integer nearest to Σ c_k g_k/2^18 - Y/2^64
//    (evaluated in units of 2^-11): with g_k = round(2^18·y_k/m_k) the
//    first term is within Σ|c_k|·2^-19 < 2^-6 of S/M, and the sum stays a
//    32-bit integer for |c_k| < m_k;
//  * L = X mod 2^64 = Σ c_k (W_k mod 2^64) - q·(M mod 2^64), exactly;
//  * H = ⌊X/2^64⌋ is the integer nearest to Y·round(M/2^51)/2^77 - L/2^64,
//    from three 32×32 products (the dropped low product is below 1 unit).
// For |c_k| < m_k the error of the estimate of X/2^64 is below 2^-3.4, so H
// is exact.  When |Y| is within about 2^52 of 2^63 (X within M/2^12 of
// ±M/2, which products bounded by Eq. M-bound never reach) the function
// returns false and the caller takes Garner's algorithm.
template <int R>
__device__ __forceinline__ bool crt_value_w64(const int (&c)[R], int E, const Oz2Moduli& mods, double& out) {
  long long y0 = 0, l0 = 0;
  uint32_t y1 = 0, l1 = 0;
  int g0 = 0;
#pragma unroll
  for (int k = 0; k < R; ++k) {
    mad_word(c[k], mods.crt_fl[k], mods.crt_fh[k], y0, y1);
    mad_word(c[k], mods.crt_wl[k], mods.crt_wh[k], l0, l1);
    g0 += c[k] * mods.crt_g[k];
  }
  const uint32_t yl = static_cast<uint32_t>(y0);
  const int yh = static_cast<int>(static_cast<uint32_t>(static_cast<u64>(y0) >> 32) + y1);
  if ((yh ^ (yh >> 31)) >= 0x7FF00000) return false;
  const int q = ((g0 >> 7) - (yh >> 21) + 1024) >> 11;
  l0 -= static_cast<long long>(q) * mods.crt_ml;
  l1 -= static_cast<uint32_t>(q) * static_cast<uint32_t>(mods.crt_mlh);
  const u64 L = static_cast<u64>(l0) + (static_cast<u64>(l1) << 32);
  const long long mid = static_cast<long long>(yh) * mods.crt_m51l +
                        static_cast<long long>(static_cast<u64>(yl) * static_cast<uint32_t>(mods.crt_m51h));
  const long long zh = static_cast<long long>(yh) * mods.crt_m51h + (mid >> 32);  // ≈ X/2^51
  const long long H = (zh - static_cast<long long>(static_cast<uint32_t>(L >> 51)) + 4096) >> 13;
  out = finish_words(H, L, E);
  return true;
}

// Fast path for r = 13 (2^112 < M < 2^121).  |X| < M/2 < 2^120, so X is
// its own residue mod 2^128 read as a signed 128-bit word, and sums that wrap
// around mod 2^128 suffice.  With u_k = c_k + coff_k ≥ 0, S = Σ u_k W_k ≡ X
// (mod M); q = ⌊S/M + 1/2⌋ comes from the 32.32 fixed-point sum
// Σ u_k F_k + 2^31 as in the five-limb path (returning false when its
// fraction is within 2^-13 of an integer, X that close to ±M/2); and
// X = (S − q·M) mod 2^128.  S mod 2^128 is formed from the word sums
// A_j = Σ u_k w_kj (w_kj the 32-bit words of W_k, j = 0..2; u_k < 2^16.1, so
// A_j < 2^52) and the top word's sum mod 2^32: four multiply-adds per
// modulus against the five-limb path's six, and no exact S.
template <int R>
__device__ __forceinline__ bool crt_value_w128(const int (&c)[R], int E, const Oz2Moduli& mods, double& out) {
  u64 a0 = 0, a1 = 0, a2 = 0;
  uint32_t a3 = 0;
  u64 Q = 1ull << 31;
#pragma unroll
  for (int k = 0; k < R; ++k) {
    const uint32_t u = static_cast<uint32_t>(c[k] + mods.coff[k]);
    a0 += static_cast<u64>(u) * mods.crtw[k][0];
    a1 += static_cast<u64>(u) * mods.crtw[k][1];
    a2 += static_cast<u64>(u) * mods.crtw[k][2];
    a3 += u * mods.crtw[k][3];
    Q += static_cast<u64>(u) * mods.crtf[k];
  }
  const uint32_t frac = static_cast<uint32_t>(Q);
  if (frac < (1u << 19) || frac > 0xFFFFFFFFu - (1u << 19)) return false;
  const u64 q = Q >> 32;
  // S mod 2^128 = hi·2^64 + lo.
  const u64 lo = a0 + (a1 << 32);
  const u64 hi = (a1 >> 32) + a2 + (static_cast<u64>(a3) << 32) + (lo < a0 ? 1ull : 0ull);
  // q·M mod 2^128 (q < 2^20).
  const u64 pl = q * mods.M[0];
  const u64 ph = q * mods.M[1] + __umul64hi(q, mods.M[0]);
  const u64 L = lo - pl;
  const u64 H = hi - ph - (lo < pl ? 1ull : 0ull);
  out = finish_words(static_cast<long long>(H), L, E);
  return true;
}

// Fast path for r = 14..16 (2^121 < M < 2^148): the same with 160-bit
// wrap-around sums, since |X| < 2^147.  S' mod 2^160 is formed from word
// sums over W_k's words 0..3 (below 2^53 for 16 moduli) and word 4's sum
// mod 2^32; q (< 2^21) and its ambiguity test are the five-limb path's.
// Five 64-bit and one 32-bit multiply-add per modulus against six 64-bit
// ones, and the subtraction of q·M and the normalisation run on three words
// instead of six limbs.
template <int R>
__device__ __forceinline__ bool crt_value_w160(const int (&c)[R], int E, const Oz2Moduli& mods, double& out) {
  u64 a0 = 0, a1 = 0, a2 = 0, a3 = 0;
  uint32_t a4 = 0;
  u64 Q = 1ull << 31;
#pragma unroll
  for (int k = 0; k < R; ++k) {
    const uint32_t u = static_cast<uint32_t>(c[k] + mods.coff[k]);
    a0 += static_cast<u64>(u) * mods.crtw[k][0];
    a1 += static_cast<u64>(u) * mods.crtw[k][1];
    a2 += static_cast<u64>(u) * mods.crtw[k][2];
    a3 += static_cast<u64>(u) * mods.crtw[k][3];
    a4 += u * mods.crtw[k][4];
    Q += static_cast<u64>(u) * mods.crtf[k];
  }
  const uint32_t frac = static_cast<uint32_t>(Q);
  if (frac < (1u << 19) || frac > 0xFFFFFFFFu - (1u << 19)) return false;
  const u64 q = Q >> 32;
  // S' mod 2^160 = top·2^128 + mid·2^64 + lo.
  const u64 lo = a0 + (a1 << 32);
  const u64 s1 = (a1 >> 32) + a2 + (lo < a0 ? 1ull : 0ull);
  const u64 mid = s1 + (a3 << 32);
  const uint32_t top = static_cast<uint32_t>(a3 >> 32) + a4 + (mid < s1 ? 1u : 0u);
  // q·M mod 2^160 (M's words 0..2 as 64-bit limbs, the last below 2^20).
  const u128 p0 = static_cast<u128>(q) * mods.M[0];
  const u128 p1 = static_cast<u128>(q) * mods.M[1] + static_cast<u64>(p0 >> 64);
  const u64 pl = static_cast<u64>(p0), pm = static_cast<u64>(p1);
  const uint32_t pt = static_cast<uint32_t>(static_cast<u64>(p1 >> 64) + q * mods.M[2]);
  u64 L = lo - pl;
  const uint32_t b0 = lo < pl ? 1u : 0u;
  u64 Mw = mid - pm - b0;
  const uint32_t b1 = (mid < pm || (mid == pm && b0)) ? 1u : 0u;
  uint32_t T = top - pt - b1;
  // Magnitude of the signed 160-bit X = T:Mw:L.
  const bool neg = (T >> 31) != 0;
  if (neg) {
    L = 0ull - L;
    const uint32_t c0 = L == 0 ? 1u : 0u;
    Mw = ~Mw + c0;
    T = ~T + ((c0 && Mw == 0) ? 1u : 0u);
  }
  // Leading 64 bits and a sticky bit for the rest.
  u64 top64;
  bool sticky;
  if (T != 0) {
    const int z = __clz(T);                      // 0..31
    const int sh = 32 - z;                       // bits of T
    top64 = (static_cast<u64>(T) << (64 - sh)) | (Mw >> sh);
    sticky = (Mw << (64 - sh)) != 0 || L != 0;
    E += 64 + sh;
  } else if (Mw != 0) {
    const int sh = 64 - __clzll(static_cast<long long>(Mw));  // 1..64
    top64 = sh == 64 ? Mw : (Mw << (64 - sh)) | (L >> sh);
    sticky = sh == 64 ? L != 0 : (L << (64 - sh)) != 0;
    E += sh;
  } else {
    top64 = L;
    sticky = false;
  }
  out = round_to_double(top64, sticky, E, neg);
  return true;
}

// 96-bit estimate for r = 11, 12 (2^102 < M < 2^112): one fixed-point sum.
// With F_k = round(2^96·y_k/m_k), Y = Σ c_k F_k mod 2^96 read as a signed
// word is 2^96·X/M + D with |D| ≤ Σ|c_k|/2, as long as that stays inside
// [-2^95, 2^95) (|Y| < 2^95 - 2^64 shows there was no wrap).  Then
// P = ⌊|Y|·M/2^96⌋, from the partial products of |Y|'s and M's 32-bit words
// at or above 2^64, is within err (a host-computed bound, about 2^27.7 for
// centred residues) of |X|, and X has Y's sign.  With P of b bits, T = P >> s
// (s = b - 64) holds P's leading 64 bits and rounds to 53 at its bit 11, so
// the midpoint between two doubles sits at bit s + 10 of P.  W, bits
// s - 21 .. s + 10 of P, puts that midpoint at bit 31; when W is more than
// e_W = ⌊err/2^(s-21)⌋ + 2 from 2^31, no midpoint lies between |X| and P,
// and the hardware conversion of T, with bit 0 set when W is above 2^31
// (T's own bits may sit exactly on the midpoint), rounds as |X| would
// (e_W < 2^29 keeps the midpoints of the binade below out of reach too).
// Returns false (the caller takes an exact path) when |Y| is too close to
// 2^95, when P < 2^85, when the test fails, or when the result would not be
// a normal double.
// The running 96-bit sum of one output: Y = a0 + a1·2^32 + a2·2^64 (mod 2^96)
// with a0, a1 exact signed 64-bit sums.
struct Y96 {
  long long a0, a1;
  uint32_t a2;
};

// Y += c·F_k for modulus k (two 32×32→64 multiply-adds and one 32-bit one).
__device__ __forceinline__ void y96_add(Y96& y, int c, const Oz2Moduli& mods, int k) {
  y.a0 += static_cast<long long>(c) * mods.crt_y0[k];
  y.a1 += static_cast<long long>(c) * mods.crt_y1[k];
  y.a2 += static_cast<uint32_t>(c) * mods.crt_y2[k];
}

__device__ __forceinline__ bool y96_finish(const Y96& y, int E, const Oz2Moduli& mods, unsigned long long err,
                                           double& out) {
  // Y as words w2:w1:w0.
  const long long s1 = (y.a0 >> 32) + y.a1;
  const uint32_t w0 = static_cast<uint32_t>(y.a0), w1 = static_cast<uint32_t>(s1);
  const uint32_t w2 = static_cast<uint32_t>(static_cast<u64>(s1) >> 32) + y.a2;
  const uint32_t sg = static_cast<uint32_t>(static_cast<int>(w2) >> 31);  // 0 or all ones
  // |Y| = (Y ^ sg) - sg
  const u64 lo = ((static_cast<u64>(w1 ^ sg) << 32) | (w0 ^ sg)) - static_cast<u64>(static_cast<long long>(static_cast<int>(sg)));
  const uint32_t y2 = (w2 ^ sg) + ((sg != 0u && lo == 0) ? 1u : 0u);
  if (y2 >= 0x7FFFFFFFu) return false;
  const uint32_t y0 = static_cast<uint32_t>(lo), y1 = static_cast<uint32_t>(lo >> 32);
  const uint32_t m0 = mods.crt_m32[0], m1 = mods.crt_m32[1], m2 = mods.crt_m32[2], m3 = mods.crt_m32[3];
  // P = Σ_{i+j≥2} y_i m_j 2^(32(i+j) - 96), the i + j = 2 products by their
  // high words: col3 (at 2^0, three products), col4 (at 2^32, two), col5
  // (at 2^64, one; m3 < 2^16).
  const u64 c2 = static_cast<u64>(__umulhi(y0, m2)) + __umulhi(y1, m1) + __umulhi(y2, m0);
  const u64 t0 = static_cast<u64>(y0) * m3 + c2;
  const u64 t1 = static_cast<u64>(y1) * m2;
  const u64 t2 = static_cast<u64>(y2) * m1;
  const u64 col4 = static_cast<u64>(y1) * m3 + static_cast<u64>(y2) * m2;
  const u64 s01 = t0 + t1;
  const u64 s012 = s01 + t2;
  const u64 pl = s012 + (col4 << 32);
  const u64 ph = static_cast<u64>(y2) * m3 + (col4 >> 32) + (s01 < t0 ? 1u : 0u) + (s012 < s01 ? 1u : 0u) +
                 (pl < s012 ? 1u : 0u);
  const int lz = __clzll(static_cast<long long>(ph));  // P has 128 - lz bits
  if (lz > 43) return false;                            // P < 2^85 (or ph = 0)
  const int sh = 64 - lz;                               // T = P >> sh, sh in [21, 48]
  const int u = sh - 21;
  const u64 ew = (err >> u) + 2;
  const uint32_t W = static_cast<uint32_t>(pl >> u);
  if (ew >= (1ull << 29) || static_cast<uint32_t>(W - 0x80000000u + static_cast<uint32_t>(ew)) <=
                                2u * static_cast<uint32_t>(ew))
    return false;
  // W ≥ 2^31 (never equal here) puts P above the midpoint of T's rounding
  // cell: bit 0 then makes a T whose low 11 bits are exactly 1024 round up.
  const u64 top = (ph << lz) | (pl >> sh) | (W >> 31);
  const int e2 = 127 - lz + E;                          // exponent of P's leading bit, scaled
  if (e2 < -1022 || e2 > 1022) return false;
  const long long bits = __double_as_longlong(__ull2double_rn(top)) + (static_cast<long long>(E + sh) << 52);
  out = __longlong_as_double(bits | (sg ? (1ll << 63) : 0ll));
  return true;
}

constexpr long long kCrtSentinel = 0x7FF4DEAD0BADF00Dll;  // a NaN the reconstruction never produces

// The reconstruction kernel's fast path by moduli count: the exact two-word
// direct CRT for r ≤ 12 (it defers only when X lies within M/2^12 of ±M/2),
// and the 128-bit and 160-bit wrap-around ones for r = 13 and r ≥ 14.
// (The 96-bit estimate above costs fewer
// multiplies but defers small and near-midpoint outputs; measured on one
// GB300 it was 3% slower at 4096³ and, on wide-range data with many small
// outputs, 20% slower, so only the fused kernel, whose per-output state must
// stay small, uses it.)
template <int R>
__device__ __forceinline__ bool crt_fast(const int (&c)[R], int E, const Oz2Moduli& mods, double& out) {
  if constexpr (R <= 12)
    return crt_value_w64<R>(c, E, mods, out);
  else if constexpr (R == 13)
    return crt_value_w128<R>(c, E, mods, out);
  else
    return crt_value_w160<R>(c, E, mods, out);
}

// The exact paths, for outputs the fast path leaves: the two-word direct CRT
// (r ≤ 12) or the five-limb one, then Garner's algorithm.
template <int R>
__device__ __noinline__ double crt_exact(const int (&c)[R], int E, const Oz2Moduli& mods) {
  double v;
  if constexpr (R <= 12) {
    if (crt_value_w64<R>(c, E, mods, v)) return v;
  } else {
    if (crt_value_fast<R>(c, E, mods, v)) return v;
  }
  return crt_value<R>(c, E, mods);
}

}  // namespace oz2
