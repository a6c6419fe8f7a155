// Residue GEMM and reconstruction fused in one tcgen05 kernel, for short k
// (§2.3 Eq. modgemm and Eq. garner; the paper's Blackwell kernel skeleton
// runs Garner in the GEMM epilogue, Algorithm 1 Phase 3): the residues of an
// output never leave the SM.  For a C with short k the r residue matrices
// (2r bytes per output, written by the residue GEMM and read back by the
// reconstruction) are the largest data the path moves; here they stay in
// registers.
//
// Work unit = one 128 × 32 output tile with every modulus.  The MMA warp
// loops over the moduli, each over all k (one K-slab: k_pad ≤ 4096 keeps
// every accumulator exact, Eq. accum-exact), into one of four accumulator
// pairs in TMEM (2 × 32 columns each), so that it runs up to three moduli
// ahead of the epilogue.  Per modulus the 16 epilogue warps read their 8
// outputs' two accumulators, release the pair, form the centred residue c_k
// (Eq. sq-shortcut / Eq. kar, as in the residue GEMM) and add c_k·F_k into the
// output's 96-bit fixed-point sum Y (the direct CRT of the reconstruction:
// Y ≈ 2^96·X/M); after the last modulus they round X·2^-(d_i+e_j) and store
// C.  The few outputs whose rounding that estimate cannot decide get a NaN
// sentinel and a place in a list; fused_fixup_kernel recomputes their
// residues from the planes and takes the exact reconstruction.  Rows and
// columns that are zero in the emulation (flag bit 1) get +0 directly.
//
// Warp 0 issues the TMA loads (a stage is one A plane tile of 128 rows and
// one B plane tile of 32 rows, 128 k-bytes each), warp 1 the MMAs
// (cta_group::1, M = 128, N = 32, K = 32), warps 2..17 the epilogue.  Every
// wait is bounded; on expiry the kernel records OZ2_ERR_TIMEOUT and drains.
//
// The 20-byte sum per output is what sizes the tile: 8 outputs per
// epilogue thread fill the registers of 16 warps, and every 32 columns of C
// then stream all of A's planes through L2 again (about 150 bytes per
// output, against the 48 bytes per output of the residue matrices' round
// trip through HBM).  The library therefore runs it only on request
// (OZ2_FLAG_FUSED).
#include "oz2_crt.cuh"
#include "oz2_gemm.cuh"

namespace oz2 {

constexpr int kFTileN = 32;                                  // output columns per tile
constexpr int kFBBytes = kFTileN * kBK;                      // B plane tile: 32 rows × 128 bytes
constexpr int kFStageBytes = kTileBytes + kFBBytes;          // 20 KiB
constexpr int kFStages = 8;
constexpr int kFBufs = 4;                                    // accumulator pairs in TMEM
constexpr int kFPairCols = 2 * kFTileN;                      // acc0, acc1 of one modulus
constexpr int kFTmemCols = kFBufs * kFPairCols;              // 256
constexpr int kFEpiWarps = 16;
constexpr int kFThreads = 32 * (2 + kFEpiWarps);
constexpr int kFCols = kFTileN / 4;                          // columns per epilogue thread
constexpr int kFixThreads = 256;
static_assert(kFStageBytes % 1024 == 0, "stages keep the 1024-byte alignment of the swizzled tiles");

struct FusedCtx {
  double* C;
  int64_t ldc;
  const int32_t* d;
  const int32_t* e;
  const uint8_t* row_flag;
  const uint8_t* col_flag;
  int* defer;            // [0]: count of outputs left; (row, col) pairs from defer + 4
  int64_t defer_cap;     // pairs the list holds
  Oz2Device* dev;
  int64_t m, n;
  unsigned long long err;
};

__device__ __forceinline__ void fused_store(const FusedCtx& ctx, int64_t row, int64_t col, const Y96& y,
                                            const Oz2Moduli& mods) {
  double v;
  if ((ctx.row_flag[row] | ctx.col_flag[col]) & 2) {
    v = 0.0;  // a zero row or column of the emulation: X = 0
  } else if (!y96_finish(y, -(ctx.d[row] + ctx.e[col]), mods, ctx.err, v)) {
    v = __longlong_as_double(kCrtSentinel);
    const int slot = atomicAdd(ctx.defer, 1);
    if (slot < ctx.defer_cap) {
      ctx.defer[4 + 2 * slot] = static_cast<int>(row);
      ctx.defer[5 + 2 * slot] = static_cast<int>(col);
    }
  }
  ctx.C[row + col * ctx.ldc] = v;
}

// SHORT1: k_pad = 128 (one k-block), whose short slab takes the
// single-correction reduction.
template <bool SHORT1>
__global__ void __launch_bounds__(kFThreads, 1)
    fused_crt_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                     const __grid_constant__ Oz2Moduli mods, int64_t k_pad, FusedCtx ctx) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kFStages * kFStageBytes);
  // bars: full[S], empty[S], acc_full[B], acc_empty[B], drain
  __shared__ uint32_t tmem_base_s;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + kFStages);
  const uint32_t accf0 = smem_u32(bars + 2 * kFStages), acce0 = smem_u32(bars + 2 * kFStages + kFBufs);
  const uint32_t drain_bar = smem_u32(bars + 2 * kFStages + 2 * kFBufs);
  const int64_t ksteps = k_pad / kBK;
  const int64_t ntm = (ctx.m + kRows - 1) / kRows, ntn = (ctx.n + kFTileN - 1) / kFTileN;
  const int64_t ntiles = ntm * ntn;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kFStages; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int b = 0; b < kFBufs; ++b) {
      mbar_init(accf0 + 8 * b, 1);
      mbar_init(acce0 + 8 * b, kFEpiWarps);
    }
    mbar_init(drain_bar, 1);
    fence_barrier_init();
    prefetch_tensormap(&tmA);
    prefetch_tensormap(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&tmem_base_s), kFTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  bool ok = true;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      uint32_t it = 0;
      for (int64_t t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
        const int64_t tm = t / ntn, tn = t - tm * ntn;
        const int64_t yb = tn * kFTileN;
        // First line of plane 0, k-block 0 of the tile's row blocks (B: its
        // 32-row part of a 128-row block; pad rows of the storage are zero).
        const int64_t la = tm * ksteps * mods.nplanes * kPlaneRows;
        const int64_t lb = (yb / kPlaneRows) * ksteps * mods.nplanes * kPlaneRows + yb % kPlaneRows;
        for (int i = 0; i < mods.r && ok; ++i) {
          const int np = mods.sq_base[i] ? 2 : 3;
          for (int64_t kb = 0; kb < ksteps && ok; ++kb) {
            for (int p = 0; p < np; ++p, ++it) {
              const int s = it % kFStages;
              if (!mbar_wait_bounded(empty0 + 8 * s, ((it / kFStages) & 1) ^ 1, kWaitLimit)) {
                ok = false;
                break;
              }
              mbar_arrive_expect_tx(full0 + 8 * s, kFStageBytes);
              const int64_t off = (kb * mods.nplanes + mods.plane_off[i] + p) * kPlaneRows;
              const uint32_t sa = smem_u32(smem + s * kFStageBytes);
              tma_load_2d(sa, &tmA, full0 + 8 * s, 0, static_cast<int>(la + off));
              tma_load_2d(sa + kTileBytes, &tmB, full0 + 8 * s, 0, static_cast<int>(lb + off));
            }
          }
        }
      }
      if (!ok) {
        ctx.dev->status = kStatusTimeout;
        ctx.dev->timeout_site = 6;
      }
      for (uint32_t j = (it > kFStages ? it - kFStages : 0); j < it; ++j)
        mbar_wait_bounded(full0 + 8 * (j % kFStages), (j / kFStages) & 1, kWaitLimit);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_f8_f32(kRows, kFTileN);
      const uint64_t desc0 = smem_desc_sw128(smem_u32(smem));
      uint32_t st = 0, ph = 0, u = 0;
      auto next = [&](uint32_t& s_, uint32_t& p_) {
        if (++s_ == kFStages) {
          s_ = 0;
          p_ ^= 1;
        }
      };
      for (int64_t t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
        for (int i = 0; i < mods.r && ok; ++i, ++u) {
          const uint32_t b = u % kFBufs;
          if (!mbar_wait_bounded(acce0 + 8 * b, ((u / kFBufs) & 1) ^ 1, kWaitLimit)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t acc0 = tmem + b * kFPairCols, acc1 = acc0 + kFTileN;
          for (int64_t kb = 0; kb < ksteps && ok; ++kb) {
            const uint32_t first = kb == 0 ? 0u : 1u;
            if (mods.sq_base[i]) {  // square: stages (d0, e0) and (d1, e1)
              uint32_t s1 = st, p1 = ph;
              next(s1, p1);
              if (!mbar_wait_bounded(full0 + 8 * st, ph, kWaitLimit) ||
                  !mbar_wait_bounded(full0 + 8 * s1, p1, kWaitLimit)) {
                ok = false;
                break;
              }
              tc_fence_after();
              const uint64_t a0 = desc0 + st * (kFStageBytes >> 4), b0 = a0 + (kTileBytes >> 4);
              const uint64_t a1 = desc0 + s1 * (kFStageBytes >> 4), b1 = a1 + (kTileBytes >> 4);
#pragma unroll
              for (int kk = 0; kk < kBK / 32; ++kk) {
                const uint32_t acc = kk ? 1u : first;
                mma_f8(acc0, a0 + 2 * kk, b0 + 2 * kk, idesc, acc);  // d0·e0
                mma_f8(acc1, a1 + 2 * kk, b0 + 2 * kk, idesc, acc);  // d1·e0
                mma_f8(acc1, a0 + 2 * kk, b1 + 2 * kk, idesc, 1u);   // + d0·e1
              }
              mma_commit(empty0 + 8 * st);
              mma_commit(empty0 + 8 * s1);
              st = s1;
              ph = p1;
              next(st, ph);
            } else {  // nonsquare: Σ·Σ → acc0; d0e0, -16 d1·e1 → acc1
              for (int p = 0; p < 3; ++p) {
                if (!mbar_wait_bounded(full0 + 8 * st, ph, kWaitLimit)) {
                  ok = false;
                  break;
                }
                tc_fence_after();
                const uint64_t a = desc0 + st * (kFStageBytes >> 4), bb = a + (kTileBytes >> 4);
#pragma unroll
                for (int kk = 0; kk < kBK / 32; ++kk) {
                  const uint32_t acc = (kk || p == 2) ? 1u : first;
                  mma_f8(p == 0 ? acc0 : acc1, a + 2 * kk, bb + 2 * kk, idesc, acc);
                }
                mma_commit(empty0 + 8 * st);
                next(st, ph);
              }
            }
          }
          if (!ok) break;
          mma_commit(accf0 + 8 * b);
        }
      }
      if (!ok) {
        ctx.dev->status = kStatusTimeout;
        ctx.dev->timeout_site = 7;
      }
      mma_commit(drain_bar);  // every MMA retired before the tensor memory goes away
      mbar_wait_bounded(drain_bar, 0, kWaitLimit);
    }
    __syncwarp();
  } else {
    // ---------------- epilogue (warps 2..17) ----------------
    const int q = warp & 3;          // TMEM lane quarter: rows 32q..32q+31 of the tile
    const int h = (warp - 2) >> 2;   // 8-column group of the tile
    const uint32_t lane_addr = tmem + (static_cast<uint32_t>(32 * q) << 16) + static_cast<uint32_t>(kFCols * h);
    uint32_t u = 0;
    for (int64_t t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
      const int64_t tm = t / ntn, tn = t - tm * ntn;
      Y96 y[kFCols];
#pragma unroll
      for (int j = 0; j < kFCols; ++j) y[j] = Y96{0, 0, 0u};
      for (int i = 0; i < mods.r; ++i, ++u) {
        const uint32_t b = u % kFBufs;
        if (!mbar_wait_bounded(accf0 + 8 * b, (u / kFBufs) & 1, kWaitLimit)) {
          ok = false;
          break;
        }
        tc_fence_after();
        uint32_t v0[kFCols], v1[kFCols];
        tmem_ld8(lane_addr + b * kFPairCols, v0);
        tmem_ld8(lane_addr + b * kFPairCols + kFTileN, v1);
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(acce0 + 8 * b);  // the pair is free for modulus i + 4
        const float mf = static_cast<float>(mods.m[i]), inv = 1.f / mf;
        const float sb = static_cast<float>(mods.sq_base[i]);
        const float hi = static_cast<float>(mods.m[i] - 1 - mods.m[i] / 2);
        if (mods.sq_base[i]) {
#pragma unroll
          for (int j = 0; j < kFCols; ++j) {
            const float r = SHORT1 ? combine_residue_short1<true>(__uint_as_float(v0[j]), __uint_as_float(v1[j]), sb,
                                                                   mf, inv, hi)
                                   : combine_residue(__uint_as_float(v0[j]), __uint_as_float(v1[j]), true, sb, mf,
                                                     inv, hi, 0.f);
            y96_add(y[j], __float_as_int(r + kRoundMagic) - 0x4B400000, mods, i);
          }
        } else {
#pragma unroll
          for (int j = 0; j < kFCols; ++j) {
            const float r = SHORT1 ? combine_residue_short1<false>(__uint_as_float(v0[j]), __uint_as_float(v1[j]), sb,
                                                                    mf, inv, hi)
                                   : combine_residue(__uint_as_float(v0[j]), __uint_as_float(v1[j]), false, sb, mf,
                                                     inv, hi, 0.f);
            y96_add(y[j], __float_as_int(r + kRoundMagic) - 0x4B400000, mods, i);
          }
        }
      }
      if (!ok) break;
      const int64_t row = tm * kRows + 32 * q + lane;
      if (row < ctx.m) {
#pragma unroll
        for (int j = 0; j < kFCols; ++j) {
          const int64_t col = tn * kFTileN + kFCols * h + j;
          if (col < ctx.n) fused_store(ctx, row, col, y[j], mods);
        }
      }
    }
    if (!ok) {
      ctx.dev->status = kStatusTimeout;
      ctx.dev->timeout_site = 8;
    }
  }
  tc_fence_before();
  __syncthreads();  // no thread leaves while MMAs or loads may touch the CTA
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, kFTmemCols);
}

// The outputs the fused kernel left, one warp each: the residues from the
// digit planes on the CUDA cores (each lane sums a strided part of k; the
// partial sums of these integer products are exact in FP32), then the exact
// reconstruction.  A list that overflowed its capacity (not possible with
// the scratch the library gives it) would leave sentinels behind.
template <int R>
__global__ void __launch_bounds__(kFixThreads)
    fused_fixup_kernel(const uint8_t* __restrict__ pa, const uint8_t* __restrict__ pb,
                       const __grid_constant__ Oz2Moduli mods, int64_t k_pad, FusedCtx ctx) {
  const int lane = threadIdx.x & 31;
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * (kFixThreads / 32);
  const int64_t count = min(static_cast<int64_t>(*ctx.defer), ctx.defer_cap);
  const int64_t kblocks = k_pad / kPlaneLine;
  for (int64_t w = (static_cast<int64_t>(blockIdx.x) * kFixThreads + threadIdx.x) / 32; w < count; w += nwarps) {
    const int64_t row = ctx.defer[4 + 2 * w], col = ctx.defer[5 + 2 * w];
    int c[R];
#pragma unroll
    for (int i = 0; i < R; ++i) {
      const bool square = mods.sq_base[i] != 0;
      float a0 = 0.f, a1 = 0.f;
      for (int64_t l = lane; l < k_pad; l += 32) {
        auto plane = [&](const uint8_t* base, int64_t rw, int j) {
          const int64_t blk = ((rw / kPlaneRows) * kblocks + l / kPlaneLine) * mods.nplanes + mods.plane_off[i] + j;
          return e4m3_to_float(base[blk * kPlaneBlock + (rw % kPlaneRows) * kPlaneLine + l % kPlaneLine]);
        };
        const float x0 = plane(pa, row, 0), y0 = plane(pb, col, 0);
        const float x1 = plane(pa, row, 1), y1 = plane(pb, col, 1);
        if (square) {
          a0 += x0 * y0;
          a1 += x1 * y0 + x0 * y1;
        } else {
          a0 += x0 * y0;
          a1 += x1 * y1 + plane(pa, row, 2) * plane(pb, col, 2);
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        a0 += __shfl_xor_sync(0xffffffffu, a0, o);
        a1 += __shfl_xor_sync(0xffffffffu, a1, o);
      }
      const float mf = static_cast<float>(mods.m[i]);
      const float r = combine_residue(a0, a1, square, static_cast<float>(mods.sq_base[i]), mf, 1.f / mf,
                                      static_cast<float>(mods.m[i] - 1 - mods.m[i] / 2), 0.f);
      c[i] = static_cast<int>(r);
    }
    if (lane == 0) ctx.C[row + col * ctx.ldc] = crt_exact<R>(c, -(ctx.d[row] + ctx.e[col]), mods);
  }
}

bool fused_crt_applies(int64_t k_pad, int r) { return (r == 11 || r == 12) && k_pad <= kFusedMaxKPad; }

static size_t fused_smem_bytes() { return 1024 + static_cast<size_t>(kFStages) * kFStageBytes + 8 * (2 * kFStages + 2 * kFBufs + 1); }

template <int R>
static cudaError_t launch_fused_r(int64_t m, int64_t n, int64_t k_pad, const Oz2Moduli& mods, const uint8_t* pa,
                                  const uint8_t* pb, const FusedCtx& ctx, cudaStream_t st) {
  CUtensorMap ta, tb;
  if (!make_block_map(&ta, pa, m, k_pad, mods.nplanes, kRows) ||
      !make_block_map(&tb, pb, n, k_pad, mods.nplanes, kFTileN))
    return cudaErrorInvalidValue;
  const size_t smem = fused_smem_bytes();
  auto kern = k_pad == kBK ? fused_crt_kernel<true> : fused_crt_kernel<false>;
  cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (err != cudaSuccess) return err;
  const int64_t ntiles = ((m + kRows - 1) / kRows) * ((n + kFTileN - 1) / kFTileN);
  const int64_t grid = std::min<int64_t>(num_sms(), ntiles);
  count_launch();
  kern<<<static_cast<unsigned>(grid), kFThreads, smem, st>>>(ta, tb, mods, k_pad, ctx);
  if ((err = cudaGetLastError()) != cudaSuccess) return err;
  count_launch();
  fused_fixup_kernel<R><<<static_cast<unsigned>(num_sms()), kFixThreads, 0, st>>>(pa, pb, mods, k_pad, ctx);
  return cudaGetLastError();
}

cudaError_t launch_fused_crt(int64_t m, int64_t n, int64_t k_pad, const Oz2Moduli& mods, const uint8_t* planes_a,
                             const uint8_t* planes_b, const int32_t* d, const int32_t* e, const uint8_t* row_flag,
                             const uint8_t* col_flag, double* C, int64_t ldc, void* scratch, size_t scratch_bytes,
                             Oz2Device* dev, cudaStream_t st) {
  if (m == 0 || n == 0) return cudaSuccess;
  if (!fused_crt_applies(k_pad, mods.r) || !scratch || reinterpret_cast<uintptr_t>(scratch) % 16 != 0 ||
      scratch_bytes < 16 + 8 * static_cast<size_t>(m) * static_cast<size_t>(n))
    return cudaErrorInvalidValue;
  FusedCtx ctx{C, ldc, d, e, row_flag, col_flag, static_cast<int*>(scratch),
               static_cast<int64_t>((scratch_bytes - 16) / 8), dev, m, n, mods.crt_err_centred};
  cudaError_t err = cudaMemsetAsync(scratch, 0, 16, st);
  if (err != cudaSuccess) return err;
  return mods.r == 11 ? launch_fused_r<11>(m, n, k_pad, mods, planes_a, planes_b, ctx, st)
                      : launch_fused_r<12>(m, n, k_pad, mods, planes_a, planes_b, ctx, st);
}

}  // namespace oz2
