// Phase 3 of Ozaki Scheme II (§2.3 Eq. garner, Appendix A; Algorithm 1
// "C ← D^-1 C̃ E^-1"): Garner mixed-radix digits per output, the integer
// X = Σ v_k P_{k-1} mapped to [-M/2, M/2), and one correctly rounded
// (round-to-nearest-even) conversion of X·2^-(d_i+e_j) to FP64, including
// the subnormal range.
//
// The reconstruction is computed by the direct CRT sum with a fixed-point
// quotient (multiply-adds only); Garner's algorithm, the paper's method,
// takes over in the rare case where that quotient is ambiguous, so every
// output equals the Garner result exactly.
//
// Residues arrive row-major (r matrices of m×n, ld = ldr ≥ n) from the
// residue GEMM; C is column-major.  A block computes a 32-row × 128-column
// tile: each thread reads four consecutive residues of one row per modulus
// (8-byte loads along n), computes its outputs, and the tile is transposed
// through shared memory so that C is written in 256-byte column segments.
#include "oz2_common.cuh"

namespace oz2 {

typedef unsigned long long u64;
typedef unsigned __int128 u128;

constexpr int kCrtRows = 32, kCrtCols = 128, kCrtThreads = 256;

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

// Fast path: the same X by the direct CRT sum.  With u_k = c_k + coff_k ≥ 0,
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

template <int R>
__global__ void __launch_bounds__(kCrtThreads) crt_kernel(int64_t m, int64_t n, const __grid_constant__ Oz2Moduli mods,
                                                          const int16_t* __restrict__ res, int64_t ldr,
                                                          const int* __restrict__ d, const int* __restrict__ e,
                                                          double* __restrict__ C, int64_t ldc, int vec_in) {
  __shared__ double tile[kCrtRows][kCrtCols + 1];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t tiles_m = static_cast<uint32_t>((m + kCrtRows - 1) / kCrtRows);
  const uint32_t ntiles = tiles_m * static_cast<uint32_t>((n + kCrtCols - 1) / kCrtCols);
  const size_t mstride = static_cast<size_t>(m) * ldr;
  for (uint32_t t = blockIdx.x; t < ntiles; t += gridDim.x) {
    const int64_t r0 = static_cast<int64_t>(t % tiles_m) * kCrtRows, c0 = static_cast<int64_t>(t / tiles_m) * kCrtCols;
    const int64_t cb = c0 + 4 * lane;
    int ecol[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) ecol[u] = cb + u < n ? e[cb + u] : 0;
    for (int s = 0; s < kCrtRows / 8; ++s) {
      const int lr = warp + 8 * s;
      const int64_t row = r0 + lr;
      if (row >= m) continue;
      const int dr = d[row];
      const int16_t* p = res + row * ldr + cb;
      uint32_t lo[R], hi[R];  // residues of columns (cb, cb+1) and (cb+2, cb+3), packed int16 pairs
      if (vec_in && cb + 3 < n) {
#pragma unroll
        for (int k = 0; k < R; ++k) {
          const uint2 q = __ldg(reinterpret_cast<const uint2*>(p + k * mstride));
          lo[k] = q.x;
          hi[k] = q.y;
        }
      } else {
#pragma unroll
        for (int k = 0; k < R; ++k) {
          uint32_t w4[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) w4[u] = cb + u < n ? static_cast<uint16_t>(p[k * mstride + u]) : 0u;
          lo[k] = w4[0] | (w4[1] << 16);
          hi[k] = w4[2] | (w4[3] << 16);
        }
      }
#pragma unroll 1
      for (int u = 0; u < 4; ++u) {
        int c[R];
#pragma unroll
        for (int k = 0; k < R; ++k) {
          const uint32_t w = u < 2 ? lo[k] : hi[k];
          c[k] = static_cast<int>(static_cast<int16_t>((u & 1) ? (w >> 16) : (w & 0xFFFFu)));
        }
        const int eu = u == 0 ? ecol[0] : u == 1 ? ecol[1] : u == 2 ? ecol[2] : ecol[3];
        double val;
        if (!crt_value_fast<R>(c, -(dr + eu), mods, val)) val = crt_value<R>(c, -(dr + eu), mods);
        tile[lr][4 * lane + u] = val;
      }
    }
    __syncthreads();
    // Column segments of 32 rows (256 bytes) per warp.
    const int64_t row = r0 + lane;
    for (int cc = warp; cc < kCrtCols; cc += kCrtThreads / 32) {
      const int64_t col = c0 + cc;
      if (col < n && row < m) C[row + col * ldc] = tile[lane][cc];
    }
    __syncthreads();
  }
}

template <int R>
static void launch_crt_r(int grid, cudaStream_t st, int64_t m, int64_t n, const Oz2Moduli& mods, const int16_t* res,
                         int64_t ldr, const int32_t* d, const int32_t* e, double* C, int64_t ldc, int vi) {
  crt_kernel<R><<<grid, kCrtThreads, 0, st>>>(m, n, mods, res, ldr, d, e, C, ldc, vi);
}

cudaError_t launch_reconstruct(int64_t m, int64_t n, const Oz2Moduli& mods, const int16_t* residues,
                               int64_t ldr, const int32_t* d, const int32_t* e, double* C, int64_t ldc,
                               cudaStream_t st) {
  if (m == 0 || n == 0) return cudaSuccess;
  const int64_t tiles = ((m + kCrtRows - 1) / kCrtRows) * ((n + kCrtCols - 1) / kCrtCols);
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int grid = static_cast<int>(tiles < 16LL * sms ? tiles : 16LL * sms);
  const int vi = (ldr % 4 == 0) && (reinterpret_cast<uintptr_t>(residues) % 8 == 0);
  count_launch();
  switch (mods.r) {
#define OZ2_CRT_CASE(R) \
  case R:               \
    launch_crt_r<R>(grid, st, m, n, mods, residues, ldr, d, e, C, ldc, vi); \
    break;
    OZ2_CRT_CASE(1) OZ2_CRT_CASE(2) OZ2_CRT_CASE(3) OZ2_CRT_CASE(4) OZ2_CRT_CASE(5) OZ2_CRT_CASE(6)
    OZ2_CRT_CASE(7) OZ2_CRT_CASE(8) OZ2_CRT_CASE(9) OZ2_CRT_CASE(10) OZ2_CRT_CASE(11) OZ2_CRT_CASE(12)
    OZ2_CRT_CASE(13) OZ2_CRT_CASE(14) OZ2_CRT_CASE(15) OZ2_CRT_CASE(16)
#undef OZ2_CRT_CASE
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace oz2
