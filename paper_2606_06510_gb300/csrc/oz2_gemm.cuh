// Definitions shared by the residue-GEMM kernels (k_gemm.cu) and the fused
// residue-GEMM + reconstruction kernel (k_fused.cu): operand tile shape,
// the mod-m epilogue arithmetic of §2.5 (Eq. sq-shortcut, Eq. kar) on the
// FMA pipe, E4M3 decoding, and the TMA descriptors of the digit planes.
#pragma once

#include <algorithm>

#include "oz2_common.cuh"

namespace oz2 {

constexpr int kRows = 128;                       // rows of an operand tile (one TMEM lane each)
constexpr int kBK = 128;                         // k-bytes per stage
constexpr int kTileBytes = kRows * kBK;          // 16 KiB
constexpr long long kWaitLimit = 4000000000LL;   // ≈2 s at 2 GHz
static_assert(kBK == kPlaneLine && kRows == kPlaneRows, "one MMA operand tile is one plane block");

// ---- epilogue arithmetic shared by the tensor-core and SIMT kernels --------
// All on the FMA pipe.  Rounding to an integer uses the 1.5·2^23 constant:
// for |y| < 2^22, fl(y + 1.5·2^23) - 1.5·2^23 = round-to-nearest(y), and the
// low 16 bits of the sum's encoding are that integer in two's complement.
constexpr float kRoundMagic = 12582912.f;  // 1.5·2^23

// x - m·round(x/m) for an exactly represented integer |x| ≤ 2^24: the FMA
// forms x - q·m exactly and q is within one of x/m, so |result| < 1.5m.
__device__ __forceinline__ float loose_mod(float x, float m, float inv_m) {
  const float q = fmaf(x, inv_m, kRoundMagic) - kRoundMagic;
  return fmaf(-q, m, x);
}
// Centred representative in [-⌊m/2⌋, m-1-⌊m/2⌋] of an integer |v| < 2^16:
// here v/m is off by under 2^-14 and lies ≥ 1/(2m) > 2^-12 from every
// half-integer unless v/m is one (even m), so the rounding is exact and only
// the tie +m/2 needs moving to -m/2.
__device__ __forceinline__ float centred_small(float v, float m, float inv_m, float hi) {
  const float q = fmaf(v, inv_m, kRoundMagic) - kRoundMagic;
  const float r = fmaf(-q, m, v);
  return r > hi ? r - m : r;
}
// Recombine one element's two accumulators (Eq. sq-shortcut, or Eq. kar with
// the merged accumulator), add the previous slab's residue, and reduce.
__device__ __forceinline__ float combine_residue(float a0, float a1, bool square, float s, float m, float inv_m,
                                                 float hi, float prev) {
  const float r0 = loose_mod(a0, m, inv_m);
  const float r1 = loose_mod(a1, m, inv_m);
  // square: d0e0 + s(d1e0 + d0e1), |v| < 2^16
  // nonsquare (b = 4): 2^b Σ + (1-2^b)(d0e0 - 2^b d1e1), |v| < 2^15
  const float v = (square ? fmaf(s, r1, r0) : fmaf(16.f, r0, -15.f * r1)) + prev;
  return centred_small(v, m, inv_m, hi);
}
// The same for a short slab, where v itself is an integer below 2^24 and the
// accumulators need no reduction before they are combined (see short_slab).
__device__ __forceinline__ float combine_residue_short(float a0, float a1, bool square, float s, float m,
                                                       float inv_m, float hi) {
  const float v = square ? fmaf(s, a1, a0) : fmaf(16.f, a0, -15.f * a1);
  return centred_small(loose_mod(v, m, inv_m), m, inv_m, hi);
}
// The short-K kernel's form (k ≤ 128, one k-block): loose_mod leaves r with
// |r| < 1.5m, so one step toward the centred range [hi + 1 - m, hi] finishes
// (above hi, r - m ≥ hi + 1 - m; below it, r + m ≤ hi), and SQUARE, uniform
// over a unit, is a template parameter.
template <bool SQUARE>
__device__ __forceinline__ float combine_residue_short1(float a0, float a1, float s, float m, float inv_m,
                                                        float hi) {
  const float v = SQUARE ? fmaf(s, a1, a0) : fmaf(16.f, a0, -15.f * a1);
  float r = loose_mod(v, m, inv_m);
  r = r > hi ? r - m : r;
  return r < hi + 1.f - m ? r + m : r;
}
// int16 encoding of an integer-valued float in [-2^15, 2^15).
__device__ __forceinline__ uint32_t as_i16_bits(float r) { return __float_as_uint(r + kRoundMagic) & 0xFFFFu; }

__device__ __forceinline__ float e4m3_to_float(uint8_t c) {
  const int e = (c >> 3) & 0xF, f = c & 7;
  float v = e ? ldexpf(static_cast<float>(8 + f), e - 10) : ldexpf(static_cast<float>(f), -9);
  return (c & 0x80) ? -v : v;
}

// ---------------------------------------------------------------------------
// Host side: tensor maps.
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

inline EncodeTiledFn get_encode_fn() {
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

// Digit planes of one operand (128 × 128-byte blocks, rows padded to 128) as
// a 2-D tensor of 128-byte lines; the box is `box_rows` lines (a whole block,
// 128, or a part of one), which land in shared memory as the tile the MMA
// descriptors expect, with the 128-byte swizzle.  Line coordinates are int32: the planes of one operand
// stay below 2^38 bytes.
inline bool make_block_map(CUtensorMap* map, const uint8_t* base, int64_t rows, int64_t k_pad, int np,
                           int box_rows = kRows) {
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) return false;
  const int64_t lines = (rows + kPlaneRows - 1) / kPlaneRows * kPlaneRows * (k_pad / kPlaneLine) * np;
  if (lines + 2 * static_cast<int64_t>(kPlaneRows) * (k_pad / kPlaneLine) * np > 0x7FFFFFFFLL) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(kPlaneLine), static_cast<cuuint64_t>(lines)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(kPlaneLine)};
  cuuint32_t box[2] = {kBK, static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

inline int num_sms() {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return sms;
}

}  // namespace oz2
