// Phase 2 of Ozaki Scheme II on FP8 tensor cores (§2.3 Eq. modgemm; §2.5
// Eq. sq-shortcut, Eq. kar, Eq. accum-exact) and the "+1" magnitude GEMM of
// §2.4, as one tcgen05 kernel for sm_103a.
//
// Per 128×128 output tile the kernel walks the moduli; per modulus it walks
// k in steps of 128 bytes (four K=32 MMAs), loading the modulus's plane
// tiles of A and B by TMA into shared memory and issuing three plane-product
// MMAs per K=32 step into FP32 accumulators in tensor memory:
//   square m = s²:  acc0 += d0·e0,  acc1 += d1·e0 + d0·e1
//   nonsquare:      acc0 += (d0+d1)(e0+e1), acc1 += d0·e0, acc2 += d1·e1
// Every K-slab (≤ 32768, Eq. accum-exact: all terms ≤ 512 so partial sums
// stay exact integers below 2^24) the epilogue warps read the accumulators,
// recombine them with the coefficients of Eq. sq-shortcut / Eq. kar, reduce
// mod m and store the centred residue as int16 (adding the previous slab's).
//
// Warp roles (192 threads): warp 0 = TMA producer, warp 1 = TMEM owner and
// MMA issuer, warps 2..5 = epilogue (warp w reads TMEM lanes 32·(w mod 4)).
// Every wait is bounded; on expiry the kernel records OZ2_ERR_TIMEOUT in the
// device status word and all roles drain and exit.
#include "oz2_common.cuh"

namespace oz2 {

constexpr int kBM = 128, kBN = 128, kBK = 128;   // tile rows, cols, k-bytes per step
constexpr int kTileBytes = kBM * kBK;            // 16 KiB per plane tile (A and B alike)
constexpr int kGemmThreads = 192;
constexpr long long kWaitLimit = 4000000000LL;   // ≈2 s at 2 GHz

template <int MODE>
struct GemmCfg;
template <>
struct GemmCfg<0> {                 // residue planes: ≤3 A and ≤3 B tiles per step
  static constexpr int kStages = 2;
  static constexpr int kMaxP = 3;
  static constexpr int kTmemCols = 512;
};
template <>
struct GemmCfg<1> {                 // magnitude plane ("+1" pass)
  static constexpr int kStages = 4;
  static constexpr int kMaxP = 1;
  static constexpr int kTmemCols = 128;
};

// ---- epilogue arithmetic shared by the tensor-core and SIMT kernels --------
// x - m·rint(x/m) for an exactly represented integer |x| < 2^24: the FMA
// forms x - q·m exactly, and q is within one of x/m, so |result| < 1.5m.
__device__ __forceinline__ float loose_mod(float x, float m, float inv_m) {
  float q = rintf(x * inv_m);
  return fmaf(-q, m, x);
}
// Centred representative in [-⌊m/2⌋, m-1-⌊m/2⌋] of an integer |x| < 2^24.
__device__ __forceinline__ int centred_mod(float x, float m, float inv_m, int lo, int hi) {
  int r = static_cast<int>(loose_mod(x, m, inv_m));
  const int mi = static_cast<int>(m);
  if (r > hi) r -= mi;
  if (r < lo) r += mi;
  if (r > hi) r -= mi;
  if (r < lo) r += mi;
  return r;
}
// Recombine one element's accumulators (Eq. sq-shortcut / Eq. kar) plus the
// previous slab's residue `prev`, and reduce.
__device__ __forceinline__ int combine_residue(float a0, float a1, float a2, bool square, float s,
                                               float m, float inv_m, int lo, int hi, int prev) {
  float r0 = loose_mod(a0, m, inv_m);
  float r1 = loose_mod(a1, m, inv_m);
  float v;
  if (square) {
    v = fmaf(s, r1, r0);                          // d0e0 + s(d1e0 + d0e1), |v| < 2^16
  } else {
    float r2 = loose_mod(a2, m, inv_m);           // 2^b Σ + (1-2^b) d0e0 + (2^2b-2^b) d1e1, b = 4
    v = fmaf(16.f, r0, fmaf(-15.f, r1, 240.f * r2));
  }
  v += static_cast<float>(prev);
  return centred_mod(v, m, inv_m, lo, hi);
}

struct EpiCtx {
  int16_t* res;        // r × (m×n, ld = m)
  float* urow;
  Oz2Device* dev;
  int64_t m, n;
};

// ---------------------------------------------------------------------------
template <int MODE>
__global__ void __launch_bounds__(kGemmThreads, 1)
    plane_gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                         const __grid_constant__ Oz2Moduli mods, int64_t k_pad, EpiCtx ctx) {
  using Cfg = GemmCfg<MODE>;
  constexpr int S = Cfg::kStages, P = Cfg::kMaxP;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;                                  // [S][P][16 KiB]
  uint8_t* sB = smem + S * P * kTileBytes;             // [S][P][16 KiB]
  uint64_t* bars = reinterpret_cast<uint64_t*>(sB + S * P * kTileBytes);
  // bars: full[S], empty[S], acc_full, acc_empty, drain
  __shared__ uint32_t tmem_base_s;
  __shared__ int abort_s;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t m0 = static_cast<int64_t>(blockIdx.x) * kBM;
  const int64_t n0 = static_cast<int64_t>(blockIdx.y) * kBN;
  const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + S);
  const uint32_t acc_full = smem_u32(bars + 2 * S), acc_empty = smem_u32(bars + 2 * S + 1);
  const uint32_t drain_bar = smem_u32(bars + 2 * S + 2);

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, 128);
    mbar_init(drain_bar, 1);
    abort_s = 0;
    fence_barrier_init();
    fence_proxy_async_smem();
    prefetch_tensormap(&tmA);
    prefetch_tensormap(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&tmem_base_s), Cfg::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;

  const int nmod = MODE == 0 ? mods.r : 1;
  const int64_t ksteps = k_pad / kBK;
  const int64_t slab_steps = MODE == 0 ? kKSlab / kBK : ksteps;
  const int64_t nslabs = (ksteps + slab_steps - 1) / slab_steps;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int i = 0; i < nmod && ok; ++i) {
        const int np = MODE == 0 ? (mods.sq_base[i] ? 2 : 3) : 1;
        const int pbase = MODE == 0 ? mods.plane_off[i] : 0;
        for (int64_t kb = 0; kb < ksteps && ok; ++kb, ++it) {
          const int s = it % S;
          const uint32_t ph = (it / S) & 1;
          if (!mbar_wait_bounded(empty0 + 8 * s, ph ^ 1, kWaitLimit) || *reinterpret_cast<volatile int*>(&abort_s)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(full0 + 8 * s, 2u * np * kTileBytes);
          for (int p = 0; p < np; ++p) {
            tma_load_3d(smem_u32(sA + (s * P + p) * kTileBytes), &tmA, full0 + 8 * s,
                        static_cast<int>(kb * kBK), static_cast<int>(m0), pbase + p);
            tma_load_3d(smem_u32(sB + (s * P + p) * kTileBytes), &tmB, full0 + 8 * s,
                        static_cast<int>(kb * kBK), static_cast<int>(n0), pbase + p);
          }
        }
      }
      if (!ok) {
        atomicExch(&abort_s, 1);
        ctx.dev->status = kStatusTimeout;
        ctx.dev->timeout_site = 1;
      }
      // Drain: wait (bounded) until every issued stage has landed.
      for (uint32_t j = (it > S ? it - S : 0); j < it; ++j)
        mbar_wait_bounded(full0 + 8 * (j % S), (j / S) & 1, kWaitLimit);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_f8_f32(kBM, kBN);
      uint32_t it = 0, accph = 0;
      bool ok = true;
      for (int i = 0; i < nmod && ok; ++i) {
        const bool square = MODE == 0 ? mods.sq_base[i] != 0 : true;
        const int np = MODE == 0 ? (square ? 2 : 3) : 1;
        for (int64_t sl = 0; sl < nslabs && ok; ++sl) {
          if (!mbar_wait_bounded(acc_empty, accph ^ 1, kWaitLimit) || *reinterpret_cast<volatile int*>(&abort_s)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const int64_t kb0 = sl * slab_steps, kb1 = min(ksteps, kb0 + slab_steps);
          for (int64_t kb = kb0; kb < kb1; ++kb, ++it) {
            const int s = it % S;
            const uint32_t ph = (it / S) & 1;
            if (!mbar_wait_bounded(full0 + 8 * s, ph, kWaitLimit) || *reinterpret_cast<volatile int*>(&abort_s)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t a0 = smem_u32(sA + (s * P) * kTileBytes);
            const uint32_t b0 = smem_u32(sB + (s * P) * kTileBytes);
#pragma unroll
            for (int kk = 0; kk < kBK / 32; ++kk) {
              const uint32_t first = (kb == kb0 && kk == 0) ? 0u : 1u;
              const uint32_t off = kk * 32;
              auto da = [&](int p) { return smem_desc_sw128(a0 + p * kTileBytes + off); };
              auto db = [&](int p) { return smem_desc_sw128(b0 + p * kTileBytes + off); };
              if (MODE == 1) {
                mma_f8(tmem, da(0), db(0), idesc, first);
              } else if (np == 2) {
                mma_f8(tmem + 0 * kBN, da(0), db(0), idesc, first);  // d0·e0
                mma_f8(tmem + 1 * kBN, da(1), db(0), idesc, first);  // d1·e0
                mma_f8(tmem + 1 * kBN, da(0), db(1), idesc, 1u);     // + d0·e1
              } else {
                mma_f8(tmem + 0 * kBN, da(0), db(0), idesc, first);  // (d0+d1)(e0+e1)
                mma_f8(tmem + 1 * kBN, da(1), db(1), idesc, first);  // d0·e0
                mma_f8(tmem + 2 * kBN, da(2), db(2), idesc, first);  // d1·e1
              }
            }
            mma_commit(empty0 + 8 * s);     // stage free once these MMAs retire
          }
          if (!ok) break;
          mma_commit(acc_full);             // accumulators complete for this slab
          accph ^= 1;
        }
      }
      if (!ok) {
        atomicExch(&abort_s, 1);
        ctx.dev->status = kStatusTimeout;
        ctx.dev->timeout_site = 2;
      }
      // Drain outstanding MMAs before the TMEM is released, through a barrier
      // of its own: an extra arrival on acc_full could complete a phase
      // beyond the one the epilogue is polling and alias its parity.
      mma_commit(drain_bar);
      mbar_wait_bounded(drain_bar, 0, kWaitLimit);
    }
    __syncwarp();
  } else {
    // ---------------- epilogue (warps 2..5) ----------------
    const int q = warp & 3;                         // TMEM lane quarter
    const int64_t row = m0 + 32 * q + lane;
    const uint32_t lane_addr = tmem + (static_cast<uint32_t>(32 * q) << 16);
    uint32_t accph = 0;
    bool ok = true;
    for (int i = 0; i < nmod && ok; ++i) {
      const bool square = MODE == 0 ? mods.sq_base[i] != 0 : true;
      const float mf = MODE == 0 ? static_cast<float>(mods.m[i]) : 1.f;
      const float inv = 1.f / mf;
      const float sb = MODE == 0 ? static_cast<float>(mods.sq_base[i]) : 0.f;
      const int lo = MODE == 0 ? -(mods.m[i] / 2) : 0;
      const int hi = MODE == 0 ? mods.m[i] - 1 - mods.m[i] / 2 : 0;
      int16_t* resi = MODE == 0 ? ctx.res + static_cast<size_t>(i) * ctx.m * ctx.n : nullptr;
      for (int64_t sl = 0; sl < nslabs; ++sl) {
        if (!mbar_wait_bounded(acc_full, accph, kWaitLimit) || *reinterpret_cast<volatile int*>(&abort_s)) {
          ok = false;
          break;
        }
        tc_fence_after();
        float rowmax = 0.f;
        for (int c = 0; c < kBN; c += 32) {
          uint32_t v0[32], v1[32], v2[32];
          tmem_ld32(lane_addr + c, v0);
          if (MODE == 0) {
            tmem_ld32(lane_addr + kBN + c, v1);
            if (!square) tmem_ld32(lane_addr + 2 * kBN + c, v2);
          }
          tmem_ld_wait();
          if (MODE == 1) {
#pragma unroll
            for (int j = 0; j < 32; ++j) rowmax = fmaxf(rowmax, __uint_as_float(v0[j]));
          } else if (row < ctx.m) {
#pragma unroll
            for (int j = 0; j < 32; ++j) {
              const int64_t col = n0 + c + j;
              if (col < ctx.n) {
                int16_t* dst = resi + col * ctx.m + row;
                const int prev = sl ? *dst : 0;
                const float a2 = square ? 0.f : __uint_as_float(v2[j]);
                *dst = static_cast<int16_t>(combine_residue(__uint_as_float(v0[j]), __uint_as_float(v1[j]),
                                                            a2, square, sb, mf, inv, lo, hi, prev));
              }
            }
          }
        }
        if (MODE == 1) {
          // rows past m hold zeros (TMA fills out-of-range rows with 0)
          if (row < ctx.m) atomicMax(reinterpret_cast<int*>(ctx.urow) + row, __float_as_int(rowmax));
          const int wm = __reduce_max_sync(0xffffffffu, __float_as_int(rowmax));
          if (lane == 0) atomicMax(&ctx.dev->u_max_bits, wm);
        }
        tc_fence_before();
        mbar_arrive(acc_empty);
        accph ^= 1;
      }
    }
    if (!ok) {
      atomicExch(&abort_s, 1);
      ctx.dev->status = kStatusTimeout;
      ctx.dev->timeout_site = 3;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, Cfg::kTmemCols);
}

// ---------------------------------------------------------------------------
// Plain CUDA-core kernel with the same semantics (diagnostic reference for
// the tensor-core path; accumulates the same integer plane products in FP32
// in sequential k order, so exactness follows from the same bound).
// ---------------------------------------------------------------------------
__device__ __forceinline__ float e4m3_to_float(uint8_t c) {
  const int e = (c >> 3) & 0xF, f = c & 7;
  float v = e ? ldexpf(static_cast<float>(8 + f), e - 10) : ldexpf(static_cast<float>(f), -9);
  return (c & 0x80) ? -v : v;
}

template <int MODE>
__global__ void plane_gemm_simt_kernel(const uint8_t* __restrict__ pa, const uint8_t* __restrict__ pb,
                                       const __grid_constant__ Oz2Moduli mods, int64_t k_pad,
                                       EpiCtx ctx) {
  const int64_t row = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const int64_t col = blockIdx.y;
  if (row >= ctx.m || col >= ctx.n) return;
  const size_t sa = static_cast<size_t>(ctx.m) * k_pad, sbs = static_cast<size_t>(ctx.n) * k_pad;
  const uint8_t* ar = pa + row * k_pad;
  const uint8_t* bc = pb + col * k_pad;
  if (MODE == 1) {
    float acc = 0.f;
    for (int64_t l = 0; l < k_pad; ++l) acc += e4m3_to_float(ar[l]) * e4m3_to_float(bc[l]);
    atomicMax(reinterpret_cast<int*>(ctx.urow) + row, __float_as_int(acc));
    atomicMax(&ctx.dev->u_max_bits, __float_as_int(acc));
    return;
  }
  for (int i = 0; i < mods.r; ++i) {
    const bool square = mods.sq_base[i] != 0;
    const float mf = static_cast<float>(mods.m[i]);
    const float inv = 1.f / mf;
    const int lo = -(mods.m[i] / 2), hi = mods.m[i] - 1 - mods.m[i] / 2;
    const size_t p0 = mods.plane_off[i];
    int res = 0;
    for (int64_t l0 = 0; l0 < k_pad; l0 += kKSlab) {
      float a0 = 0.f, a1 = 0.f, a2 = 0.f;
      const int64_t l1 = min(k_pad, l0 + kKSlab);
      for (int64_t l = l0; l < l1; ++l) {
        const float x0 = e4m3_to_float(ar[p0 * sa + l]), y0 = e4m3_to_float(bc[p0 * sbs + l]);
        const float x1 = e4m3_to_float(ar[(p0 + 1) * sa + l]), y1 = e4m3_to_float(bc[(p0 + 1) * sbs + l]);
        if (square) {
          a0 += x0 * y0;
          a1 += x1 * y0 + x0 * y1;
        } else {
          const float x2 = e4m3_to_float(ar[(p0 + 2) * sa + l]), y2 = e4m3_to_float(bc[(p0 + 2) * sbs + l]);
          a0 += x0 * y0;
          a1 += x1 * y1;
          a2 += x2 * y2;
        }
      }
      res = combine_residue(a0, a1, a2, square, static_cast<float>(mods.sq_base[i]), mf, inv, lo, hi, res);
    }
    ctx.res[static_cast<size_t>(i) * ctx.m * ctx.n + col * ctx.m + row] = static_cast<int16_t>(res);
  }
}

// ---------------------------------------------------------------------------
// Host side: tensor maps and launch.
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// Planes of one operand: `np` planes of rows × k_pad bytes, row-major.
static bool make_plane_map(CUtensorMap* map, const uint8_t* base, int64_t rows, int64_t k_pad, int np) {
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(k_pad), static_cast<cuuint64_t>(rows),
                        static_cast<cuuint64_t>(np)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(k_pad), static_cast<cuuint64_t>(rows * k_pad)};
  cuuint32_t box[3] = {kBK, static_cast<cuuint32_t>(kBM), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<uint8_t*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <int MODE>
static size_t gemm_smem_bytes() {
  using Cfg = GemmCfg<MODE>;
  return 1024 + 2 * static_cast<size_t>(Cfg::kStages) * Cfg::kMaxP * kTileBytes + 8 * (2 * Cfg::kStages + 3);
}

// mode: 0 residues (tensor cores), 1 magnitude (tensor cores),
//       2 residues (SIMT reference), 3 magnitude (SIMT reference).
cudaError_t launch_plane_gemm(int64_t m, int64_t n, int64_t k_pad, const Oz2Moduli& mods,
                              const uint8_t* planes_a, const uint8_t* planes_b, int mode,
                              int16_t* residues, float* urow, Oz2Device* dev, cudaStream_t st) {
  if (m == 0 || n == 0) return cudaSuccess;
  EpiCtx ctx{residues, urow, dev, m, n};
  if (mode >= 2) {
    dim3 g(static_cast<unsigned>((m + 127) / 128), static_cast<unsigned>(n));
    count_launch();
    if (mode == 2) plane_gemm_simt_kernel<0><<<g, 128, 0, st>>>(planes_a, planes_b, mods, k_pad, ctx);
    else plane_gemm_simt_kernel<1><<<g, 128, 0, st>>>(planes_a, planes_b, mods, k_pad, ctx);
    return cudaGetLastError();
  }
  const int np = mode == 0 ? mods.nplanes : 1;
  CUtensorMap ta, tb;
  if (!make_plane_map(&ta, planes_a, m, k_pad, np) || !make_plane_map(&tb, planes_b, n, k_pad, np))
    return cudaErrorInvalidValue;
  dim3 g(static_cast<unsigned>((m + kBM - 1) / kBM), static_cast<unsigned>((n + kBN - 1) / kBN));
  cudaError_t err;
  if (mode == 0) {
    size_t smem = gemm_smem_bytes<0>();
    if ((err = cudaFuncSetAttribute(plane_gemm_tc_kernel<0>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    static_cast<int>(smem))) != cudaSuccess)
      return err;
    count_launch();
    plane_gemm_tc_kernel<0><<<g, kGemmThreads, smem, st>>>(ta, tb, mods, k_pad, ctx);
  } else {
    size_t smem = gemm_smem_bytes<1>();
    if ((err = cudaFuncSetAttribute(plane_gemm_tc_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    static_cast<int>(smem))) != cudaSuccess)
      return err;
    count_launch();
    plane_gemm_tc_kernel<1><<<g, kGemmThreads, smem, st>>>(ta, tb, mods, k_pad, ctx);
  }
  return cudaGetLastError();
}

}  // namespace oz2
