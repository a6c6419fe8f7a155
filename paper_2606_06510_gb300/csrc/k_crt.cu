// Phase 3 of Ozaki Scheme II (§2.3 Eq. garner, Appendix A; Algorithm 1
// "C ← D^-1 C̃ E^-1"): the integer X ∈ [-M/2, M/2) with the given residues
// and one correctly rounded (round-to-nearest-even) conversion of
// X·2^-(d_i+e_j) to FP64, including the subnormal range.
//
// X is computed by the direct CRT sum in fixed point (multiply-adds only):
// an exact two-word sum for r ≤ 12 and 128- and 160-bit wrap-around sums
// for r = 13 and r ≥ 14, with
// Garner's algorithm, the paper's method, taking over in the rare case where
// that sum's quotient is ambiguous.  Every output equals the Garner result
// exactly.
//
// Residues arrive column-major (r matrices of m×n, ld = ldr ≥ m) from the
// residue GEMM and C is column-major, so a thread takes two consecutive
// rows of a column: one 4-byte load per modulus (a warp reads 128 bytes per
// modulus) and one 16-byte store of its two results (a warp writes 512
// contiguous bytes), with no transposition.  Each thread walks a strided
// set of columns and loads the next column's residues while it computes the
// current one.  An output that the fast path leaves is recorded in a short
// per-thread list (local memory, touched only then) and recomputed after the
// loop, which keeps the exact paths' registers out of the loop; past the
// list's length the output is marked with a NaN sentinel and found again by
// a rescan of the thread's later columns.
#include "oz2_crt.cuh"

namespace oz2 {

constexpr int kCrtThreads = 256;
constexpr int kCrtFailSlots = 8;  // outputs per thread the fast path may leave before a rescan

// Resident blocks per SM the register budget is sized for: the two-word
// path fits 64 registers (four blocks) up to r = 12 in the FAST kernel and
// up to r = 10 in the element-wise one; the 128-bit path (r = 13) 80 (three
// blocks); the 160-bit path (r ≥ 14) takes 128 (at 80 it spills and ran
// 13 to 41% slower).
template <int R, bool FAST>
constexpr int crt_min_blocks() {
  return R <= (FAST ? 12 : 10) ? 4 : (R <= 13 ? 3 : 2);
}

// The columns of one thread (two rows, or one at an odd last row): each
// column's residues are loaded while the previous column is reconstructed,
// alternating between two buffers.  FAST: both rows present, 4-byte residue
// loads and 16-byte stores possible; otherwise element-wise accesses.
// Outputs the fast path leaves go into `fails` as 2·(column iteration) + row
// (0 or 1), the first kCrtFailSlots of them; returns how many there were.
template <int R, bool FAST>
__device__ __forceinline__ int crt_columns(int64_t n, int64_t row, bool pair, int d0, int d1, const Oz2Moduli& mods,
                                           const int16_t* __restrict__ res, int64_t ldr, const int* __restrict__ e,
                                           double* cbase, int64_t ldc, int (&fails)[kCrtFailSlots]) {
  const int64_t step = gridDim.y;
  const int64_t off_step = step * ldr;
  // Residue matrix k starts at res + k·mstride (the same for every thread,
  // formed once); this thread's entry of a column is row + col·ldr elements
  // further.
  const size_t mstride = static_cast<size_t>(n) * ldr;
  const int16_t* base[R];
#pragma unroll
  for (int k = 0; k < R; ++k) base[k] = res + k * mstride;
  // Two rows' residues of one column, packed (row in the low half).
  auto load_words = [&](int64_t off, uint32_t (&w)[R]) {
    if (FAST) {
#pragma unroll
      for (int k = 0; k < R; ++k) w[k] = __ldg(reinterpret_cast<const uint32_t*>(base[k] + off));
    } else {
#pragma unroll
      for (int k = 0; k < R; ++k)
        w[k] = static_cast<uint16_t>(base[k][off]) | (pair ? static_cast<uint32_t>(base[k][off + 1]) << 16 : 0u);
    }
  };
  int nfail = 0;
  int iter = 0;
  auto column = [&](const uint32_t (&w)[R], int ec, int64_t col) {
    double v[2];
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      int c[R];
#pragma unroll
      for (int k = 0; k < R; ++k)
        c[k] = u ? (static_cast<int>(w[k]) >> 16) : static_cast<int>(static_cast<int16_t>(w[k] & 0xFFFFu));
      double val;
      if (!crt_fast<R>(c, -((u ? d1 : d0) + ec), mods, val)) {
        val = __longlong_as_double(kCrtSentinel);
        if (nfail < kCrtFailSlots) fails[nfail] = 2 * iter + u;
        ++nfail;
      }
      v[u] = val;
    }
    ++iter;
    double* out = cbase + col * ldc;
    if (FAST) {
      *reinterpret_cast<double2*>(out) = make_double2(v[0], v[1]);
    } else {
      out[0] = v[0];
      if (pair) out[1] = v[1];
    }
  };
  uint32_t wa[R], wb[R];
  int ea = 0, eb = 0;
  int64_t col = blockIdx.y, off = col * ldr + row;
  if (col < n) {
    load_words(off, wa);
    ea = __ldg(e + col);
  }
  while (col < n) {
    if (col + step < n) {
      load_words(off + off_step, wb);
      eb = __ldg(e + col + step);
    }
    column(wa, ea, col);
    col += step;
    off += off_step;
    if (col >= n) break;
    if (col + step < n) {
      load_words(off + off_step, wa);
      ea = __ldg(e + col + step);
    }
    column(wb, eb, col);
    col += step;
    off += off_step;
  }
  return nfail;
}

// Rows [row0, row0 + rows) of C.  FAST kernels take row pairs with 4-byte
// residue loads and 16-byte stores (rows even, residues and C aligned); the
// other kernel takes any rows element-wise.  The two are separate kernels so
// that each gets its own register allocation.
template <int R, bool FAST>
__global__ void __launch_bounds__(kCrtThreads, crt_min_blocks<R, FAST>())
    crt_kernel(int64_t row0, int64_t rows, int64_t n, const __grid_constant__ Oz2Moduli mods,
               const int16_t* __restrict__ res, int64_t ldr, const int* __restrict__ d, const int* __restrict__ e,
               double* __restrict__ C, int64_t ldc) {
  const int64_t rel = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) * 2;
  if (rel >= rows) return;
  const int64_t row = row0 + rel;
  const bool pair = rel + 1 < rows;
  const int d0 = d[row], d1 = pair ? d[row + 1] : 0;
  double* cbase = C + row;
  int fails[kCrtFailSlots];
  const int nfail = crt_columns<R, FAST>(n, row, pair, d0, d1, mods, res, ldr, e, cbase, ldc, fails);
  if (nfail == 0) return;
  // Outputs the fast path left to the exact paths (this thread's own).
  const int64_t step = gridDim.y;
  auto exact = [&](int64_t col, int u) {
    int c[R];
#pragma unroll
    for (int k = 0; k < R; ++k) c[k] = res[(k * n + col) * ldr + row + u];
    cbase[col * ldc + u] = crt_exact<R>(c, -((u ? d1 : d0) + __ldg(e + col)), mods);
  };
  const int listed = nfail < kCrtFailSlots ? nfail : kCrtFailSlots;
  for (int i = 0; i < listed; ++i) exact(blockIdx.y + (fails[i] >> 1) * step, fails[i] & 1);
  if (nfail > kCrtFailSlots) {
    // More than the list holds: the rest carry the sentinel, from the column
    // of the last one listed on (whose other row may be one of them).
    for (int64_t col = blockIdx.y + (fails[kCrtFailSlots - 1] >> 1) * step; col < n; col += step)
      for (int u = 0; u < (pair ? 2 : 1); ++u)
        if (__double_as_longlong(cbase[col * ldc + u]) == kCrtSentinel) exact(col, u);
  }
}

// One launch over rows [row0, row0 + rows): x covers row pairs, y strides
// over the columns, about two waves of resident blocks in all.
template <int R, bool FAST>
static cudaError_t launch_crt_rows(cudaStream_t st, int64_t row0, int64_t rows, int64_t n, const Oz2Moduli& mods,
                                   const int16_t* res, int64_t ldr, const int32_t* d, const int32_t* e, double* C,
                                   int64_t ldc) {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t gx = ((rows + 1) / 2 + kCrtThreads - 1) / kCrtThreads;
  if (gx > 0x7FFFFFFF) return cudaErrorInvalidValue;
  int64_t gy = (2LL * crt_min_blocks<R, FAST>() * sms + gx - 1) / gx;
  gy = gy < 1 ? 1 : gy;
  gy = gy > n ? n : gy;
  gy = gy > 65535 ? 65535 : gy;
  count_launch();
  crt_kernel<R, FAST><<<dim3(static_cast<unsigned>(gx), static_cast<unsigned>(gy)), kCrtThreads, 0, st>>>(
      row0, rows, n, mods, res, ldr, d, e, C, ldc);
  return cudaGetLastError();
}

template <int R>
static cudaError_t launch_crt_r(cudaStream_t st, int64_t m, int64_t n, const Oz2Moduli& mods, const int16_t* res,
                                int64_t ldr, const int32_t* d, const int32_t* e, double* C, int64_t ldc) {
  const bool vec = (ldr % 2 == 0) && (reinterpret_cast<uintptr_t>(res) % 4 == 0) && (ldc % 2 == 0) &&
                   (reinterpret_cast<uintptr_t>(C) % 16 == 0);
  if (!vec) return launch_crt_rows<R, false>(st, 0, m, n, mods, res, ldr, d, e, C, ldc);
  const int64_t even = m & ~int64_t{1};
  cudaError_t err = cudaSuccess;
  if (even > 0) err = launch_crt_rows<R, true>(st, 0, even, n, mods, res, ldr, d, e, C, ldc);
  if (err == cudaSuccess && even < m)
    err = launch_crt_rows<R, false>(st, even, 1, n, mods, res, ldr, d, e, C, ldc);
  return err;
}

cudaError_t launch_reconstruct(int64_t m, int64_t n, const Oz2Moduli& mods, const int16_t* residues,
                               int64_t ldr, const int32_t* d, const int32_t* e, double* C, int64_t ldc,
                               cudaStream_t st) {
  if (m == 0 || n == 0) return cudaSuccess;
  switch (mods.r) {
#define OZ2_CRT_CASE(R) \
  case R:               \
    return launch_crt_r<R>(st, m, n, mods, residues, ldr, d, e, C, ldc);
    OZ2_CRT_CASE(1) OZ2_CRT_CASE(2) OZ2_CRT_CASE(3) OZ2_CRT_CASE(4) OZ2_CRT_CASE(5) OZ2_CRT_CASE(6)
    OZ2_CRT_CASE(7) OZ2_CRT_CASE(8) OZ2_CRT_CASE(9) OZ2_CRT_CASE(10) OZ2_CRT_CASE(11) OZ2_CRT_CASE(12)
    OZ2_CRT_CASE(13) OZ2_CRT_CASE(14) OZ2_CRT_CASE(15) OZ2_CRT_CASE(16)
#undef OZ2_CRT_CASE
    default:
      return cudaErrorInvalidValue;
  }
}

}  // namespace oz2
