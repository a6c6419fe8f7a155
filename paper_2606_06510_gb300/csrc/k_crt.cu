// Phase 3 of Ozaki Scheme II (§2.3 Eq. garner, Appendix A; Algorithm 1
// "C ← D^-1 C̃ E^-1"): Garner mixed-radix digits per output, the integer
// X = Σ v_k P_{k-1} mapped to [-M/2, M/2), and one correctly rounded
// (round-to-nearest-even) conversion of X·2^-(d_i+e_j) to FP64, including
// the subnormal range.
#include "oz2_common.cuh"

namespace oz2 {

typedef unsigned long long u64;
typedef unsigned int u32;

// X (3 limbs, little-endian) = X·m + v.
__device__ __forceinline__ void mul_add(u64 (&x)[3], uint32_t m, uint32_t v, bool three) {
  u64 lo = x[0] * m;
  u64 c = __umul64hi(x[0], m);
  u64 s0 = lo + v;
  c += s0 < lo;
  u64 l1 = x[1] * m;
  u64 c1 = __umul64hi(x[1], m);
  u64 s1 = l1 + c;
  c1 += s1 < l1;
  x[0] = s0;
  x[1] = s1;
  if (three) x[2] = x[2] * m + c1;
}

__device__ __forceinline__ bool geq3(const u64 (&a)[3], const u64 (&b)[3]) {
  if (a[2] != b[2]) return a[2] > b[2];
  if (a[1] != b[1]) return a[1] > b[1];
  return a[0] >= b[0];
}

__device__ __forceinline__ void sub3(const u64 (&a)[3], const u64 (&b)[3], u64 (&r)[3]) {
  u64 r0 = a[0] - b[0];
  u64 br = a[0] < b[0];
  u64 t1 = a[1] - b[1];
  u64 br1 = a[1] < b[1];
  u64 r1 = t1 - br;
  br1 |= t1 < br;
  r[0] = r0;
  r[1] = r1;
  r[2] = a[2] - b[2] - br1;
}

__device__ __forceinline__ int bitlen3(const u64 (&x)[3]) {
  if (x[2]) return 192 - __clzll(static_cast<long long>(x[2]));
  if (x[1]) return 128 - __clzll(static_cast<long long>(x[1]));
  if (x[0]) return 64 - __clzll(static_cast<long long>(x[0]));
  return 0;
}

// `cnt` (≤ 64) bits of x starting at bit `pos` (pos ≥ 0).
__device__ __forceinline__ u64 bits3(const u64 (&x)[3], int pos, int cnt) {
  const int w = pos >> 6, b = pos & 63;
  u64 lo = w < 3 ? x[w] : 0;
  u64 hi = w + 1 < 3 ? x[w + 1] : 0;
  u64 v = b ? (lo >> b) | (hi << (64 - b)) : lo;
  return cnt >= 64 ? v : (v & ((1ull << cnt) - 1));
}

// Any bit of x below position pos (pos ≥ 0)?
__device__ __forceinline__ bool sticky3(const u64 (&x)[3], int pos) {
  if (pos <= 0) return false;
  const int w = pos >> 6, b = pos & 63;
  bool s = false;
  for (int t = 0; t < 3 && t < w; ++t) s |= x[t] != 0;
  if (w < 3 && b) s |= (x[w] & ((1ull << b) - 1)) != 0;
  return s;
}

// Nearest double (ties to even) to (-1)^neg · mag · 2^E.
__device__ __forceinline__ double round_to_double(const u64 (&mag)[3], int E, bool neg) {
  const int L = bitlen3(mag);
  const u64 sign = neg ? (1ull << 63) : 0ull;
  if (L == 0) return __longlong_as_double(static_cast<long long>(sign));
  const int top = L - 1 + E;                     // exponent of the leading bit
  if (top > 1023) return __longlong_as_double(static_cast<long long>(sign | 0x7FF0000000000000ull));
  const int p = top >= -1022 ? 53 : top + 1075;  // significant bits available
  const int sh = L - p;                          // bits dropped (may be ≤ 0)
  u64 q;
  if (sh <= 0) {
    q = mag[0] << (-sh);                         // L ≤ 53: exact
  } else if (p <= 0) {
    // Everything is below the last subnormal bit position + 1.
    const bool above_half = (p == 0) && sticky3(mag, L - 1);  // mag > 2^(L-1) = half
    q = above_half ? 1 : 0;
  } else {
    q = bits3(mag, sh, p);
    const bool rbit = bits3(mag, sh - 1, 1) != 0;
    const bool st = sticky3(mag, sh - 1);
    if (rbit && (st || (q & 1))) ++q;
  }
  if (q == 0) return __longlong_as_double(static_cast<long long>(sign));
  if (p < 53 || top < -1022) {
    // Subnormal scale: value = q · 2^-1074 (q = 2^52 is the smallest normal).
    return __longlong_as_double(static_cast<long long>(sign | q));
  }
  int f = top;                                   // q ∈ [2^52, 2^53]
  if (q >> 53) {
    q >>= 1;
    ++f;
  }
  if (f > 1023) return __longlong_as_double(static_cast<long long>(sign | 0x7FF0000000000000ull));
  const u64 bits = (static_cast<u64>(f + 1023) << 52) | (q & ((1ull << 52) - 1));
  return __longlong_as_double(static_cast<long long>(sign | bits));
}

// One output: centred residues c[0..R) → nearest double of X·2^E.
template <int R>
__device__ __forceinline__ double crt_value(const int (&c)[R], int E, const Oz2Moduli& mods) {
  // Garner digits (Eq. garner): v_k = (c_k - Σ_{j<k} v_j P_{j-1}) P_{k-1}^{-1} mod m_k,
  // with (P_{j-1} mod m_k) precomputed; goff_k (a multiple of m_k ≥ 2^27) keeps
  // the 32-bit sum positive.
  uint32_t v[R];
#pragma unroll
  for (int k = 0; k < R; ++k) {
    int acc = mods.goff[k] + c[k];
#pragma unroll
    for (int t = 0; t < k; ++t) acc -= static_cast<int>(v[t]) * mods.pmod[k][t];
    const uint32_t mk = static_cast<uint32_t>(mods.m[k]);
    const uint32_t t0 = mod_magic(static_cast<uint32_t>(acc), mk, mods.magic[k], mods.magic_sh[k]);
    v[k] = mod_magic(t0 * static_cast<uint32_t>(mods.inv[k]), mk, mods.magic[k], mods.magic_sh[k]);
  }
  // Mixed radix → integer by Horner from the top digit.  The top six digits
  // stay below 2^61 (six moduli ≤ 1089), so they run in 64-bit arithmetic.
  constexpr int H = R < 6 ? R : 6;
  u64 top = v[R - 1];
#pragma unroll
  for (int k = R - 2; k >= R - H; --k) top = top * static_cast<u32>(mods.m[k]) + v[k];
  u64 X[3] = {top, 0, 0};
#pragma unroll
  for (int k = R - H - 1; k >= 0; --k) mul_add(X, static_cast<uint32_t>(mods.m[k]), v[k], R > 12);
  // Symmetric range [-M/2, M/2) (Eq. M-bound): X ≥ ⌈M/2⌉ ⇔ 2X ≥ M.
  const bool neg = geq3(X, mods.Mhalf);
  u64 mag[3];
  if (neg) {
    sub3(mods.M, X, mag);
  } else {
    mag[0] = X[0];
    mag[1] = X[1];
    mag[2] = X[2];
  }
  return round_to_double(mag, E, neg);
}

// Four consecutive rows of one column per thread: 8-byte residue loads per
// modulus (int16 × 4) and two 16-byte stores of C when the layout allows.
// The four outputs are computed one after the other (not interleaved) to keep
// the register footprint of the r-deep Garner recurrence small.
template <int R>
__global__ void __launch_bounds__(256) crt_kernel(int64_t m, int64_t n, const __grid_constant__ Oz2Moduli mods,
                                                  const int16_t* __restrict__ res, int64_t ldr,
                                                  const int* __restrict__ d, const int* __restrict__ e,
                                                  double* __restrict__ C, int64_t ldc, int vec_in, int vec_out) {
  const int64_t i0 = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) * 4;
  if (i0 >= m) return;
  const bool full = i0 + 3 < m;
  const size_t mstride = static_cast<size_t>(ldr) * n;
  int di[4];
#pragma unroll
  for (int u = 0; u < 4; ++u) di[u] = i0 + u < m ? d[i0 + u] : 0;
  for (int64_t j = blockIdx.y; j < n; j += gridDim.y) {
    const int16_t* p = res + j * ldr + i0;
    uint32_t lo[R], hi[R];   // residues of rows (i0, i0+1) and (i0+2, i0+3), packed int16 pairs
    if (vec_in && full) {
#pragma unroll
      for (int k = 0; k < R; ++k) {
        const uint2 q = __ldg(reinterpret_cast<const uint2*>(p + k * mstride));
        lo[k] = q.x;
        hi[k] = q.y;
      }
    } else {
#pragma unroll
      for (int k = 0; k < R; ++k) {
        uint32_t w[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) w[u] = i0 + u < m ? static_cast<uint16_t>(p[k * mstride + u]) : 0u;
        lo[k] = w[0] | (w[1] << 16);
        hi[k] = w[2] | (w[3] << 16);
      }
    }
    const int ej = e[j];
    double2 o01, o23;
#pragma unroll 1
    for (int u = 0; u < 4; ++u) {
      int c[R];
#pragma unroll
      for (int k = 0; k < R; ++k) {
        const uint32_t w = u < 2 ? lo[k] : hi[k];
        c[k] = static_cast<int>(static_cast<int16_t>((u & 1) ? (w >> 16) : (w & 0xFFFFu)));
      }
      const int du = u == 0 ? di[0] : u == 1 ? di[1] : u == 2 ? di[2] : di[3];
      const double val = crt_value<R>(c, -(du + ej), mods);
      if (u == 0) o01.x = val;
      else if (u == 1) o01.y = val;
      else if (u == 2) o23.x = val;
      else o23.y = val;
    }
    double* q = C + i0 + j * ldc;
    if (vec_out && full) {
      reinterpret_cast<double2*>(q)[0] = o01;
      reinterpret_cast<double2*>(q)[1] = o23;
    } else {
      const double out[4] = {o01.x, o01.y, o23.x, o23.y};
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (i0 + u < m) q[u] = out[u];
    }
  }
}

template <int R>
static void launch_crt_r(dim3 g, cudaStream_t st, int64_t m, int64_t n, const Oz2Moduli& mods, const int16_t* res,
                         int64_t ldr, const int32_t* d, const int32_t* e, double* C, int64_t ldc, int vi, int vo) {
  crt_kernel<R><<<g, 256, 0, st>>>(m, n, mods, res, ldr, d, e, C, ldc, vi, vo);
}

cudaError_t launch_reconstruct(int64_t m, int64_t n, const Oz2Moduli& mods, const int16_t* residues,
                               int64_t ldr, const int32_t* d, const int32_t* e, double* C, int64_t ldc,
                               cudaStream_t st) {
  if (m == 0 || n == 0) return cudaSuccess;
  dim3 g(static_cast<unsigned>((m + 1023) / 1024), static_cast<unsigned>(n < 65535 ? n : 65535));
  const int vi = (ldr % 4 == 0) && (reinterpret_cast<uintptr_t>(residues) % 8 == 0);
  const int vo = (ldc % 2 == 0) && (reinterpret_cast<uintptr_t>(C) % 16 == 0);
  count_launch();
  switch (mods.r) {
#define OZ2_CRT_CASE(R) \
  case R:               \
    launch_crt_r<R>(g, st, m, n, mods, residues, ldr, d, e, C, ldc, vi, vo); \
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
