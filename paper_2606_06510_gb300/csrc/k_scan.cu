// Phase 1 of Ozaki Scheme II (§2.3 Eq. scale; Algorithm 1 "scan the exponent
// spans of A, B; choose power-of-two diagonals D, E"): the exponent scan, the
// fallback flags, and the choice of D and E from the "+1" pass (§2.4).
#include <climits>

#include "k_scan.cuh"

namespace oz2 {

// Scan key of one element: 0 for zero, (frexp exponent + 2048) for a finite
// nonzero value (frexp exponent e: |x| = f·2^e, f ∈ [0.5, 1), so |x| < 2^e),
// and 1<<20 for Inf/NaN.  The max over a row is therefore the max-exponent
// of its finite entries, unless the row holds a non-finite value.
__device__ __forceinline__ int scan_key(double x) {
  unsigned long long b = __double_as_longlong(x);
  int E = static_cast<int>((b >> 52) & 0x7FF);
  unsigned long long mant = b & ((1ull << 52) - 1);
  if (E == 0x7FF) return 1 << 20;
  if (E == 0) {
    if (mant == 0) return 0;
    int bl = 64 - __clzll(static_cast<long long>(mant));  // bit length of the subnormal significand
    return bl - 1074 + 2048;
  }
  return E - 1022 + 2048;
}

// Rows of column-major A: thread per row, block row `by` of the k-chunks.
__device__ __forceinline__ void scan_a_rows(int64_t bx, int64_t by, int64_t m, int64_t k,
                                            const double* __restrict__ A, int64_t lda, int chunk,
                                            int* __restrict__ key) {
  int64_t i = bx * (int64_t)blockDim.x + threadIdx.x;
  if (i >= m) return;
  int64_t l0 = by * chunk;
  int64_t l1 = min(k, l0 + chunk);
  int best = 0;
  const double* p = A + i + l0 * lda;
  int64_t l = l0;
  for (; l + 4 <= l1; l += 4, p += 4 * lda) {
    double x0 = __ldg(p), x1 = __ldg(p + lda), x2 = __ldg(p + 2 * lda), x3 = __ldg(p + 3 * lda);
    best = max(best, max(max(scan_key(x0), scan_key(x1)), max(scan_key(x2), scan_key(x3))));
  }
  for (; l < l1; ++l, p += lda) best = max(best, scan_key(__ldg(p)));
  if (best) atomicMax(key + i, best);
}

// Columns of column-major B: warp per column, lanes over l, block row `by`
// of the even-sized k-chunks; 16-byte loads when the column start is aligned.
__device__ __forceinline__ void scan_b_cols(int64_t bx, int64_t by, int64_t n, int64_t k,
                                            const double* __restrict__ B, int64_t ldb, int chunk, int vec,
                                            int* __restrict__ key) {
  int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int64_t j = bx * (int64_t)(blockDim.x >> 5) + warp;
  if (j >= n) return;
  int64_t l0 = by * chunk;
  int64_t l1 = min(k, l0 + chunk);
  const double* col = B + j * ldb;
  int best = 0;
  if (vec) {
    const double2* c2 = reinterpret_cast<const double2*>(col);
    const int64_t p1 = l1 >> 1;  // pairs fully inside [l0, l1) (l0 is even)
    int64_t p = (l0 >> 1) + lane;
    for (; p + 96 < p1; p += 128) {
      const double2 a = __ldg(c2 + p), b = __ldg(c2 + p + 32), c = __ldg(c2 + p + 64), d = __ldg(c2 + p + 96);
      best = max(best, max(max(max(scan_key(a.x), scan_key(a.y)), max(scan_key(b.x), scan_key(b.y))),
                           max(max(scan_key(c.x), scan_key(c.y)), max(scan_key(d.x), scan_key(d.y)))));
    }
    for (; p < p1; p += 32) {
      const double2 a = __ldg(c2 + p);
      best = max(best, max(scan_key(a.x), scan_key(a.y)));
    }
    if ((l1 & 1) && lane == 0) best = max(best, scan_key(__ldg(col + l1 - 1)));
  } else {
    int64_t l = l0 + lane;
    for (; l + 96 < l1; l += 128)
      best = max(best, max(max(scan_key(__ldg(col + l)), scan_key(__ldg(col + l + 32))),
                           max(scan_key(__ldg(col + l + 64)), scan_key(__ldg(col + l + 96)))));
    for (; l < l1; l += 32) best = max(best, scan_key(__ldg(col + l)));
  }
  best = __reduce_max_sync(0xffffffffu, best);
  if (lane == 0 && best) atomicMax(key + j, best);
}

// Both operands in one launch: blocks [0, ga) scan rows of A (gax blocks of
// 256 rows per k-chunk), the rest scan columns of B (gbx blocks of 8 columns
// per k-chunk).
struct ScanGrid {
  int64_t ga, gax, gbx;
  int achunk, bchunk, vec;
};
__global__ void __launch_bounds__(256) scan_kernel(int64_t m, int64_t n, int64_t k, const double* __restrict__ A,
                                                   int64_t lda, const double* __restrict__ B, int64_t ldb, ScanGrid g,
                                                   int* __restrict__ ra, int* __restrict__ cb) {
  pdl_trigger();  // the flags kernel may be scheduled now; it waits for this grid to finish
  const int64_t b = blockIdx.x;
  if (b < g.ga) {
    scan_a_rows(b % g.gax, b / g.gax, m, k, A, lda, g.achunk, ra);
  } else {
    const int64_t bb = b - g.ga;
    scan_b_cols(bb % g.gbx, bb / g.gbx, n, k, B, ldb, g.bchunk, g.vec, cb);
  }
}

// One block per operand (block b takes operand first_op + b; 0: rows of A,
// 1: columns of B).  Decodes the scan keys, finds the lower median of the exponents of the nonzero finite rows,
// and writes the flags (bit0: native fallback; bit1: zero in the emulation)
// and the final exponent (0 for rows that are zero in the emulation).
constexpr int kExpBins = 2112;   // frexp exponents of finite doubles: [-1073, 1024]
constexpr int kExpBias = 1080;
constexpr int kFinalizeThreads = 1024;
constexpr int kBinsPerThread = (kExpBins + kFinalizeThreads - 1) / kFinalizeThreads;

__global__ void __launch_bounds__(kFinalizeThreads) finalize_flags_kernel(int64_t m, int64_t n, int* __restrict__ ra,
                                      int* __restrict__ cb, uint8_t* __restrict__ row_flag,
                                      uint8_t* __restrict__ col_flag, unsigned flags,
                                      Oz2Device* dev, int first_op) {
  __shared__ int hist[kExpBins];
  __shared__ int warp_sum[32];
  __shared__ int med_s;
  __shared__ int count_s;
  pdl_wait();  // the scan keys are complete
  const bool is_a = blockIdx.x + first_op == 0;
  const int64_t cnt = is_a ? m : n;
  int* key = is_a ? ra : cb;
  uint8_t* fl = is_a ? row_flag : col_flag;
  for (int b = threadIdx.x; b < kExpBins; b += blockDim.x) hist[b] = 0;
  if (threadIdx.x == 0) count_s = 0;
  __syncthreads();
  for (int64_t i = threadIdx.x; i < cnt; i += blockDim.x) {
    int kv = key[i];
    if (kv > 0 && kv < (1 << 20)) atomicAdd(&hist[kv - 2048 + kExpBias], 1);
  }
  __syncthreads();
  // Lower median of the histogram: each thread sums kBinsPerThread bins, a
  // block-wide inclusive scan of those sums locates the bin that holds the
  // element of rank ⌊(total-1)/2⌋.
  {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const int b0 = threadIdx.x * kBinsPerThread;
    int mine = 0;
#pragma unroll
    for (int j = 0; j < kBinsPerThread; ++j) mine += b0 + j < kExpBins ? hist[b0 + j] : 0;
    int incl = mine;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    if (lane == 31) warp_sum[wid] = incl;
    __syncthreads();
    if (wid == 0) {
      int w = lane < kFinalizeThreads / 32 ? warp_sum[lane] : 0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, w, o);
        if (lane >= o) w += v;
      }
      warp_sum[lane] = w;  // inclusive prefix over warps
    }
    __syncthreads();
    incl += wid ? warp_sum[wid - 1] : 0;
    const int total = warp_sum[kFinalizeThreads / 32 - 1];
    if (threadIdx.x == 0) med_s = 0;
    __syncthreads();
    if (total > 0) {
      const int rank = (total - 1) / 2;
      int acc = incl - mine;  // exclusive prefix
      if (acc <= rank && rank < incl) {
        for (int j = 0; j < kBinsPerThread; ++j) {
          acc += hist[b0 + j];
          if (acc > rank) {
            med_s = b0 + j - kExpBias;
            break;
          }
        }
      }
    }
    __syncthreads();
  }
  const int med = med_s;
  const bool window = (flags & OZ2_FLAG_NO_FALLBACK) == 0;
  int local = 0;
  for (int64_t i = threadIdx.x; i < cnt; i += blockDim.x) {
    int kv = key[i];
    bool nonfinite = kv >= (1 << 20);
    bool nonzero = kv > 0 && !nonfinite;
    int e = nonzero ? kv - 2048 : 0;
    bool fb = nonfinite || (window && nonzero && abs(e - med) > kFallbackWindow);
    bool zero = fb || !nonzero;
    fl[i] = static_cast<uint8_t>((fb ? 1 : 0) | (zero ? 2 : 0));
    key[i] = zero ? 0 : e;
    local += fb ? 1 : 0;
  }
  if (local) atomicAdd(&count_s, local);
  __syncthreads();
  if (threadIdx.x == 0 && dev) {
    if (is_a) dev->fallback_rows = count_s;
    else dev->fallback_cols = count_s;
  }
}

cudaError_t launch_scan_keys(int64_t m, int64_t n, int64_t k, const double* A, int64_t lda, const double* B,
                             int64_t ldb, ScanOut out, cudaStream_t st) {
  if (k <= 0 || (m <= 0 && n <= 0)) return cudaSuccess;
  ScanGrid g{};
  g.achunk = 64;
  int64_t ks = (k + g.achunk - 1) / g.achunk;
  if (ks > 65535) {
    g.achunk = static_cast<int>((k + 65534) / 65535);
    ks = (k + g.achunk - 1) / g.achunk;
  }
  g.bchunk = 1024;
  int64_t bks = (k + g.bchunk - 1) / g.bchunk;
  if (bks > 65535) {
    g.bchunk = static_cast<int>((k + 65534) / 65535 + 1) & ~1;
    bks = (k + g.bchunk - 1) / g.bchunk;
  }
  g.gax = (m + 255) / 256;
  g.ga = m > 0 ? g.gax * ks : 0;
  g.gbx = (n + 7) / 8;
  const int64_t gb = n > 0 ? g.gbx * bks : 0;
  g.vec = (ldb % 2 == 0) && (reinterpret_cast<uintptr_t>(B) % 16 == 0);
  if (g.ga + gb > 0x7FFFFFFFLL) return cudaErrorInvalidValue;
  count_launch();
  scan_kernel<<<static_cast<unsigned>(g.ga + gb), 256, 0, st>>>(m, n, k, A, lda, B, ldb, g, out.ra, out.cb);
  return cudaGetLastError();
}

cudaError_t launch_scan_flags(int64_t m, int64_t n, int ops, unsigned flags, ScanOut out, Oz2Device* dev,
                              cudaStream_t st) {
  if ((ops & 3) == 0) return cudaSuccess;
  const int first = (ops & 1) ? 0 : 1;
  const int count = ops == 3 ? 2 : 1;
  count_launch();
  const cudaError_t e = launch_dependent(finalize_flags_kernel, dim3(count), dim3(kFinalizeThreads), 0, st, m, n,
                                         out.ra, out.cb, out.row_flag, out.col_flag, flags, dev, first);
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_scan(int64_t m, int64_t n, int64_t k, const double* A, int64_t lda,
                        const double* B, int64_t ldb, unsigned flags, ScanOut out,
                        Oz2Device* dev, cudaStream_t st, bool zero_keys) {
  cudaError_t err;
  // The scan keys are maxima taken with atomics: zero unless the caller has.
  if (zero_keys && m > 0 && (err = cudaMemsetAsync(out.ra, 0, sizeof(int) * m, st)) != cudaSuccess) return err;
  if (zero_keys && n > 0 && (err = cudaMemsetAsync(out.cb, 0, sizeof(int) * n, st)) != cudaSuccess) return err;
  if ((err = launch_scan_keys(m, n, k, A, lda, B, ldb, out, st)) != cudaSuccess) return err;
  return launch_scan_flags(m, n, 3, flags, out, dev, st);
}

// ---------------------------------------------------------------------------
// Scale choice (reading R-scale of the "+1" pass, or the crude bound R1).
// ---------------------------------------------------------------------------
// ⌈log2 U⌉ of a positive normal float.
__device__ __forceinline__ int ceil_log2_f32(float u) {
  unsigned b = __float_as_uint(u);
  int E = static_cast<int>((b >> 23) & 0xFF);
  return E - 127 + ((b & 0x7FFFFFu) ? 1 : 0);
}

__global__ void choose_scales_kernel(int64_t m, int64_t n, int64_t k, int T, int scale_mode,
                                     const float* __restrict__ urow, const int* __restrict__ ra,
                                     const int* __restrict__ cb,
                                     const uint8_t* __restrict__ row_flag,
                                     const uint8_t* __restrict__ col_flag, int* __restrict__ d,
                                     int* __restrict__ e, Oz2Device* dev) {
  int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  int s, umax = 0;
  if (scale_mode == OZ2_SCALE_R2) {
    float ug = __int_as_float(dev->u_max_bits);
    umax = ug > 0.f ? ceil_log2_f32(ug) : 0;
    s = min(62, (T - umax) >> 1);
  } else {
    int lk = k <= 1 ? 0 : 64 - __clzll(static_cast<long long>(k - 1));
    int pA = min(62, (T - lk) >> 1);
    s = min(62, T - lk - pA);
    if (idx < m) {
      d[idx] = (row_flag[idx] & 2) ? 0 : pA - ra[idx];
    } else if (idx < m + n) {
      int64_t j = idx - m;
      e[j] = (col_flag[j] & 2) ? 0 : s - cb[j];
    }
    if (idx == 0) dev->s = s;
    return;
  }
  if (idx < m) {
    float u = urow[idx];
    int ui = u > 0.f ? ceil_log2_f32(u) : umax;
    int t = min(62, T - s - ui);
    d[idx] = (row_flag[idx] & 2) ? 0 : t - ra[idx];
  } else if (idx < m + n) {
    int64_t j = idx - m;
    e[j] = (col_flag[j] & 2) ? 0 : s - cb[j];
  }
  if (idx == 0) dev->s = s;
}

cudaError_t launch_choose_scales(int64_t m, int64_t n, int64_t k, const Oz2Moduli& mods,
                                 int scale_mode, const float* urow, const int32_t* ra,
                                 const int32_t* cb, const uint8_t* row_flag,
                                 const uint8_t* col_flag, int32_t* d, int32_t* e,
                                 Oz2Device* dev, cudaStream_t st) {
  int64_t tot = m + n;
  if (tot == 0) return cudaSuccess;
  count_launch();
  choose_scales_kernel<<<static_cast<unsigned>((tot + 255) / 256), 256, 0, st>>>(
      m, n, k, mods.T, scale_mode, urow, ra, cb, row_flag, col_flag, d, e, dev);
  return cudaGetLastError();
}

}  // namespace oz2
