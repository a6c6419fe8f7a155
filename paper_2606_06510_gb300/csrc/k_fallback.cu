// Native-FP64 fallback (Algorithm 1, the "if" on admissibility; §2.6 contract
// item (vi)): rows of A (columns of B) flagged by the scan are recomputed
// with FP64 FMA chains, every output C_ij = fma(A_i,k-1, B_k-1,j, ... fma(A_i0,
// B_0j, +0)), in the order l = 0..k-1, so the result is reproducible.
//
// Tiled CUDA-core DGEMM over index lists: 64×64 output tiles, 256 threads,
// 4×4 outputs per thread, k staged through shared memory in chunks of 16.
// The same kernel is the cuBLAS-free native comparator (identity lists).
#include <algorithm>

#include "oz2_common.cuh"

namespace oz2 {

constexpr int kFT = 64, kFK = 16;

// Compact the rows (blockIdx.y = 0) and columns (blockIdx.y = 1) whose flag
// has bit0 set into their lists, counting in count[0] and count[1].
__global__ void compact_flags_kernel(int64_t m, int64_t n, const uint8_t* __restrict__ row_flag,
                                     const uint8_t* __restrict__ col_flag, int* __restrict__ row_list,
                                     int* __restrict__ col_list, int* __restrict__ count) {
  const bool cols = blockIdx.y == 1;
  const int64_t cnt = cols ? n : m;
  const uint8_t* flag = cols ? col_flag : row_flag;
  int* list = cols ? col_list : row_list;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < cnt; i += (int64_t)gridDim.x * blockDim.x)
    if (flag[i] & 1) list[atomicAdd(count + (cols ? 1 : 0), 1)] = static_cast<int>(i);
}

// rows: row_list ? row_list[0..*row_count) : 0..m-1 ; cols likewise.  With
// gridDim.y = 2 the blocks with blockIdx.y = 0 take the row list against all
// columns and those with blockIdx.y = 1 all rows against the column list.
__global__ void __launch_bounds__(256) fma_gemm_kernel(int64_t m, int64_t n, int64_t k,
                                                       const double* __restrict__ A, int64_t lda,
                                                       const double* __restrict__ B, int64_t ldb,
                                                       const int* __restrict__ row_list,
                                                       const int* __restrict__ row_count,
                                                       const int* __restrict__ col_list,
                                                       const int* __restrict__ col_count, double* __restrict__ C,
                                                       int64_t ldc) {
  __shared__ double As[kFK][kFT + 1];
  __shared__ double Bs[kFK][kFT + 1];
  __shared__ int rid[kFT], cid[kFT];
  if (gridDim.y == 2) {
    if (blockIdx.y == 0) {
      col_list = nullptr;
    } else {
      row_list = nullptr;
    }
  }
  const int64_t nr = row_list ? *row_count : m;
  const int64_t nc = col_list ? *col_count : n;
  const int64_t rt = (nr + kFT - 1) / kFT, ct = (nc + kFT - 1) / kFT;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  for (int64_t tile = blockIdx.x; tile < rt * ct; tile += gridDim.x) {
    const int64_t r0 = (tile % rt) * kFT, c0 = (tile / rt) * kFT;
    __syncthreads();
    if (threadIdx.x < kFT) {
      const int64_t a = r0 + threadIdx.x;
      rid[threadIdx.x] = a < nr ? (row_list ? row_list[a] : static_cast<int>(a)) : -1;
    } else if (threadIdx.x < 2 * kFT) {
      const int64_t b = c0 + threadIdx.x - kFT;
      cid[threadIdx.x - kFT] = b < nc ? (col_list ? col_list[b] : static_cast<int>(b)) : -1;
    }
    __syncthreads();
    double acc[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) acc[a][b] = 0.0;
    for (int64_t l0 = 0; l0 < k; l0 += kFK) {
      __syncthreads();
      // A tile: 64 rows × 16 k; thread loads 4 entries (row = t % 64, k = t / 64 + 4q).
      for (int q = 0; q < 4; ++q) {
        const int rr = threadIdx.x & 63, kk = (threadIdx.x >> 6) + 4 * q;
        const int gi = rid[rr];
        const int64_t l = l0 + kk;
        As[kk][rr] = (gi >= 0 && l < k) ? A[gi + l * lda] : 0.0;
        const int cc = threadIdx.x & 63;
        const int gj = cid[cc];
        // B tile: 16 k × 64 cols; same pattern (k fastest would coalesce better;
        // the fallback is rare and small).
        Bs[kk][cc] = (gj >= 0 && l < k) ? B[l + gj * ldb] : 0.0;
      }
      __syncthreads();
      const int kmax = static_cast<int>(k - l0 < kFK ? k - l0 : kFK);
      for (int kk = 0; kk < kmax; ++kk) {
        double av[4], bv[4];
#pragma unroll
        for (int a = 0; a < 4; ++a) av[a] = As[kk][ty * 4 + a];
#pragma unroll
        for (int b = 0; b < 4; ++b) bv[b] = Bs[kk][tx * 4 + b];
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
          for (int b = 0; b < 4; ++b) acc[a][b] = fma(av[a], bv[b], acc[a][b]);
      }
    }
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      const int gi = rid[ty * 4 + a];
      if (gi < 0) continue;
#pragma unroll
      for (int b = 0; b < 4; ++b) {
        const int gj = cid[tx * 4 + b];
        if (gj >= 0) C[gi + static_cast<int64_t>(gj) * ldc] = acc[a][b];
      }
    }
  }
}

static int fb_grid() {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return sms * 4;
}

// scratch: (m + n + 2) ints of device memory (counts, then the lists); the
// two counts must be zero on entry unless `zero_counts` is set.
cudaError_t launch_fallback_lists(int64_t m, int64_t n, int64_t k, const double* A, int64_t lda, const double* B,
                                  int64_t ldb, const uint8_t* row_flag, const uint8_t* col_flag, int* scratch,
                                  double* C, int64_t ldc, cudaStream_t st, bool zero_counts) {
  if (m == 0 || n == 0) return cudaSuccess;
  int* counts = scratch;              // [0]: rows, [1]: cols
  int* rlist = scratch + 2;
  int* clist = rlist + m;
  if (zero_counts) {
    const cudaError_t err = cudaMemsetAsync(counts, 0, 2 * sizeof(int), st);
    if (err != cudaSuccess) return err;
  }
  count_launch(2);
  const int64_t most = m > n ? m : n;
  const unsigned cg = static_cast<unsigned>(std::min<int64_t>((most + 255) / 256, 4096));
  compact_flags_kernel<<<dim3(cg, 2), 256, 0, st>>>(m, n, row_flag, col_flag, rlist, clist, counts);
  // flagged rows × all columns (blockIdx.y = 0), all rows × flagged columns (1)
  fma_gemm_kernel<<<dim3(fb_grid(), 2), 256, 0, st>>>(m, n, k, A, lda, B, ldb, rlist, counts, clist, counts + 1, C,
                                                       ldc);
  return cudaGetLastError();
}

cudaError_t launch_native(int64_t m, int64_t n, int64_t k, const double* A, int64_t lda, const double* B,
                          int64_t ldb, double* C, int64_t ldc, cudaStream_t st) {
  if (m == 0 || n == 0) return cudaSuccess;
  count_launch();
  fma_gemm_kernel<<<fb_grid(), 256, 0, st>>>(m, n, k, A, lda, B, ldb, nullptr, nullptr, nullptr, nullptr, C, ldc);
  return cudaGetLastError();
}

}  // namespace oz2
