// Deconstruction (Algorithm 1 "lin:quant" and "lin:dec"; §2.5 digit planes)
// and the magnitude planes of the "+1" pass (§2.4).
//
// One thread handles 8 consecutive k-entries of one row of the operand (a row
// of A, or a column of B seen as a row of Bᵀ).  In the deconstruction, 16
// threads share a row and cover 128 consecutive k-entries, so each plane row
// segment they write is one full 128-byte line (8-byte stores per thread);
// partial lines written by different blocks at different times cost the
// memory system a read-modify-write each.  The magnitude pass writes one
// plane only and is faster with 4 threads per row (32-byte segments, more
// rows in flight per block).  A is column-major: the threads of a warp that
// load the same k-entries read consecutive rows.  B's rows are contiguous in
// k and are read with 16-byte vector loads.  One launch covers both
// operands: the first blocks work on A, the rest on B.
#include <algorithm>
#include <utility>

#include "oz2_gemm.cuh"

namespace oz2 {

constexpr int kElems = 8;  // k-entries per thread

// Launch and tile shape of each pass: threads per block, resident blocks per
// SM (64 registers a thread either way), threads per row, k-entries per tile
// column (a divisor of the k padding) and rows per block.  The
// deconstruction's blocks are large so that two of them, each with its own
// copy of the digit-plane table, fill an SM.
template <int MODE>
struct TileShape {
  static constexpr int kThreads = MODE == 0 ? 256 : 512;
  static constexpr int kBlocksPerSm = MODE == 0 ? 8 : 2;
  static constexpr int kThreadsPerRow = MODE == 0 ? 4 : 16;
  static constexpr int kSeg = kElems * kThreadsPerRow;
  static constexpr int kRows = kThreads / kThreadsPerRow;
};
static_assert(kKPad % TileShape<0>::kSeg == 0 && kKPad % TileShape<1>::kSeg == 0, "tile column must divide k_pad");
static_assert(TileShape<1>::kSeg == kPlaneLine, "a row's threads write whole plane lines");

// Integer significand M and exponent x with |x| = M·2^x (M < 2^53), or M = 0.
struct Split {
  unsigned long long M;
  int ex;
  bool neg;
};
__device__ __forceinline__ Split split_double(double v) {
  unsigned long long b = __double_as_longlong(v);
  Split s;
  s.neg = (b >> 63) != 0;
  int E = static_cast<int>((b >> 52) & 0x7FF);
  unsigned long long mant = b & ((1ull << 52) - 1);
  if (E == 0x7FF) {  // non-finite entries only occur in rows zeroed by the flags
    s.M = 0;
    s.ex = 0;
  } else if (E == 0) {
    s.M = mant;
    s.ex = -1074;
  } else {
    s.M = mant | (1ull << 52);
    s.ex = E - 1075;
  }
  return s;
}

// ⌊2^d |v|⌉ (TZ: toward zero, RN: half to even) as an unsigned integer; the
// scale choice guarantees the result is below 2^62.
__device__ __forceinline__ unsigned long long quantise_abs(const Split& s, int d, bool rn) {
  if (s.M == 0) return 0;
  int sh = s.ex + d;
  if (sh >= 0) return s.M << min(sh, 63);
  int r = -sh;
  if (r >= 64) return 0;  // < 2^53·2^-64 < 1/2
  unsigned long long q = s.M >> r;
  if (rn) {
    unsigned long long rem = s.M & ((1ull << r) - 1);
    unsigned long long half = 1ull << (r - 1);
    if (rem > half || (rem == half && (q & 1))) ++q;
  }
  return q;
}

// The 21-bit limbs of 8 integer entries Ã (|Ã| < 2^62) as the residue sums
// take them: w0 = v0 + kDecBias (bits 0-20 plus the bias), w1 = v1 (bits
// 21-41) and w2 = v2 (bits 42-63, signed).
struct Limbs {
  uint32_t w0[kElems];
  uint32_t w1[kElems];
  int w2[kElems];
};

// Entry e of L from Ã as a two's complement word (tl: bits 0-31, th: 32-63).
__device__ __forceinline__ void set_limbs(Limbs& L, int e, uint32_t tl, int th) {
  L.w0[e] = (tl & ((1u << kLimbBits) - 1)) | kDecBias;
  L.w1[e] = __funnelshift_r(tl, static_cast<uint32_t>(th), kLimbBits) & ((1u << kLimbBits) - 1);
  L.w2[e] = th >> (2 * kLimbBits - 32);
}

// Truncating quantisation (Eq. scale, TZ) of entry e: Ã = trunc(x·2^d) as
// a 64-bit two's complement word, for rows with d ≤ kTzFastMaxD, into the
// limbs L.  With x = ±M·2^(sh - d), M < 2^53, Ã = ±⌊M·2^10 / 2^(10 - sh)⌋: the
// significand is shifted up by 10 (below 2^63) and then right by r = 10 - sh
// with clamping funnel shifts, so zeros, subnormals and entries that shift
// out entirely need no branch.  That needs sh ≤ 9: a normal x has M ≥ 2^52
// and |Ã| < 2^62, and a subnormal one has sh = d - 1074 ≤ 9 for
// d ≤ kTzFastMaxD (rows with a larger scale, whose largest entry is itself
// subnormal, take the general path).  d = -4096 gives Ã = 0 for any x.
constexpr int kTzFastMaxD = 1083;
__device__ __forceinline__ void quantise_tz_limbs(double x, int d, Limbs& L, int e) {
  const uint32_t hi = static_cast<uint32_t>(__double2hiint(x)), lo = static_cast<uint32_t>(__double2loint(x));
  const int E = static_cast<int>((hi >> 20) & 0x7FFu);
  const uint32_t mh = (hi & 0xFFFFFu) | (E ? 0x100000u : 0u);  // M = mh·2^32 + lo
  const uint32_t r = static_cast<uint32_t>(10 + 1075 - max(E, 1) - d);
  const uint32_t ph = __funnelshift_l(lo, mh, 10), pl = lo << 10;  // M·2^10
  const bool wide = r >= 32;
  const uint32_t x1 = wide ? 0u : ph, x0 = wide ? ph : pl, rr = wide ? r - 32 : r;
  const uint32_t al = __funnelshift_rc(x0, x1, rr), ah = __funnelshift_rc(x1, 0u, rr);
  const uint32_t sgn = static_cast<uint32_t>(static_cast<int>(hi) >> 31);  // 0 or all ones
  const unsigned long long t = ((static_cast<unsigned long long>(ah ^ sgn) << 32) | (al ^ sgn)) -
                               static_cast<unsigned long long>(static_cast<long long>(static_cast<int>(sgn)));
  set_limbs(L, e, static_cast<uint32_t>(t), static_cast<int>(t >> 32));
}

// ⌈log2 |v|⌉ for finite nonzero v.
__device__ __forceinline__ int ceil_log2_abs(const Split& s) {
  int bl = 64 - __clzll(static_cast<long long>(s.M));
  bool pow2 = (s.M & (s.M - 1)) == 0;
  return s.ex + (pow2 ? bl - 1 : bl);
}

// E4M3 code of 2^q, q ∈ [-9, 0] (subnormal below 2^-6).
__device__ __forceinline__ uint32_t e4m3_pow2(int q) {
  return q >= -6 ? static_cast<uint32_t>((q + 7) << 3) : (1u << (q + 9));
}

// Magnitude-plane code of x: 0 for x = 0, else the E4M3 code of
// 2^max(-c, ⌈log2|x|⌉ - ex).  A normal double has ⌈log2|x|⌉ = E - 1023, plus
// one when its fraction is nonzero, read off the high word; subnormals take
// the general path.
__device__ __forceinline__ uint32_t magnitude_code(double x, int ex, int c) {
  const unsigned long long b = __double_as_longlong(x);
  const uint32_t hi = static_cast<uint32_t>(b >> 32), lo = static_cast<uint32_t>(b);
  const int E = static_cast<int>((hi >> 20) & 0x7FFu);
  const bool frac = ((hi & 0xFFFFFu) | lo) != 0;
  if (E == 0x7FF) return 0u;  // non-finite entries only occur in rows zeroed by the flags
  if (E == 0) {
    if (!frac) return 0u;
    const Split sp = split_double(x);
    return e4m3_pow2(max(-c, ceil_log2_abs(sp) - ex));
  }
  return e4m3_pow2(max(-c, E - 1023 + (frac ? 1 : 0) - ex));
}

// Rows a pass writes: the magnitude plane has the operand's rows, the digit
// planes whole 128-row blocks.
template <int MODE>
__host__ __device__ __forceinline__ int64_t rows_stored(int64_t rows) {
  return MODE == 0 ? rows : (rows + kPlaneRows - 1) / kPlaneRows * kPlaneRows;
}

// Bytes 0, 1 and 2 of four 32-bit words w0..w3 gathered into p0, p1, p2
// (byte j of p_b is byte b of w_j): a 4 × 4 byte transpose in two rounds of
// byte permutes, seven in all.
__device__ __forceinline__ void transpose3(uint32_t w0, uint32_t w1, uint32_t w2, uint32_t w3, uint32_t& p0,
                                           uint32_t& p1, uint32_t& p2) {
  const uint32_t t0 = __byte_perm(w0, w1, 0x5140), t1 = __byte_perm(w0, w1, 0x7362);  // w0.b0 w1.b0 w0.b1 w1.b1 | .b2 .b3
  const uint32_t t2 = __byte_perm(w2, w3, 0x5140), t3 = __byte_perm(w2, w3, 0x7362);
  p0 = __byte_perm(t0, t2, 0x5410);
  p1 = __byte_perm(t0, t2, 0x7632);
  p2 = __byte_perm(t1, t3, 0x5410);
}

struct OperandView {
  const double* base;
  int64_t row_stride;   // A: 1, B: ldb
  int64_t k_stride;     // A: lda, B: 1
  int64_t rows;
  const int32_t* exps;  // ra/cb (magnitude) or d/e (deconstruction)
  const uint8_t* flag;
  uint8_t* out;         // planes: rows × k_pad per plane
  const uint32_t* table;  // packed digit planes per residue (deconstruction)
  int vec;              // k contiguous and rows 16-byte aligned: vector loads
};

// The 8 entries [l0, l0+8) of one row (zero beyond k).
__device__ __forceinline__ void load8(const OperandView& X, int64_t row, int64_t l0, int64_t k, double (&x)[kElems]) {
  const double* p = X.base + row * X.row_stride + l0 * X.k_stride;
  if (X.vec && l0 + kElems <= k) {
#pragma unroll
    for (int t = 0; t < kElems / 2; ++t) {
      const double2 v = __ldg(reinterpret_cast<const double2*>(p) + t);
      x[2 * t] = v.x;
      x[2 * t + 1] = v.y;
    }
  } else {
#pragma unroll
    for (int e = 0; e < kElems; ++e) x[e] = l0 + e < k ? __ldg(p + e * X.k_stride) : 0.0;
  }
}

// Residues of 8 entries modulo modulus I and their E4M3 digit planes (the
// modulus's constants are compile-time constants).
//
// Y = w0 + w1·c1 + w2·c2 (32-bit wrap-around; the true value lies in
// (0, 2^32)) is congruent to Ã + kDecBias mod m.  With magic = ⌈2^32/m⌉,
// q = ⌊Y·magic/2^32⌋ = ⌊Y/m + Y·(magic·m - 2^32)/(m·2^32)⌋ is ⌊Y/m⌋ or one
// more, since the second term is below Y/2^32 < 1; so Y - qm lies in
// [-m, m) and indexes a table whose 2m entries start m entries before it,
// rotated by the bias.
// E4M3 codes of two integer-valued floats, `lo` in bits 0-7 and `hi` in
// bits 8-15 (exact: both are integers of magnitude at most 16).
__device__ __forceinline__ uint32_t e4m3x2(float lo, float hi) {
  uint16_t r;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(hi), "f"(lo));
  return r;
}
// The integer v (|v| < 2^22) as a float: 1.5·2^23 + v has ulp 1.
__device__ __forceinline__ float small_int_float(uint32_t biased) {
  return __int_as_float(static_cast<int>(biased)) - 12582912.0f;
}

// Square modulus m = s² (§2.5, balanced base s): the digits of the centred
// residue c are computed, not looked up.  With u = c + h0 + s·h1 ≥ 0,
// d0 = (u mod s) - h0 and d1 = ⌊u/s⌋ - h1.  u = ((Y + E) mod m) + h0 + s·h1 -
// ⌊m/2⌋, since c = ((x + ⌊m/2⌋) mod m) - ⌊m/2⌋ for x = Ã mod m = (Y - B)
// mod m.  (Y + E) mod m comes from the same magic quotient as the table
// index, corrected once.
// Plane j of modulus I lands at dst + (plane_off(I) + j - PBASE)·STRIDE: the
// block layout in global memory (STRIDE = one 16 KiB block, PBASE 0), or the
// operand tiles of the on-the-fly kernel in shared memory.
template <int I, int STRIDE = kPlaneBlock, int PBASE = 0>
__device__ __forceinline__ void square_digits(const Limbs& L, uint8_t* dst) {
  constexpr ModConst mc = mod_const(I);
  constexpr int kShift = mc.sq_h0 + mc.s * mc.sq_h1 - mc.m / 2;  // u - (Y + E) mod m, ≥ 0
  float f0[kElems], f1[kElems];
#pragma unroll
  for (int e = 0; e < kElems; ++e) {
    const uint32_t Y = L.w0[e] + mc.sq_e + L.w1[e] * static_cast<uint32_t>(mc.c1) +
                       static_cast<uint32_t>(L.w2[e]) * static_cast<uint32_t>(mc.c2);
    const uint32_t q = __umulhi(Y, mc.magic);
    int off = static_cast<int>(Y - q * static_cast<uint32_t>(mc.m));  // (Y mod m) or that - m
    off += off < 0 ? mc.m : 0;
    if constexpr (mc.s == 32) {
      const uint32_t u = static_cast<uint32_t>(off) + kShift;
      f0[e] = small_int_float((u & 31u) + (0x4B400000u - mc.sq_h0));
      f1[e] = small_int_float((u >> 5) + (0x4B400000u - mc.sq_h1));
    } else {
      // u = off + kShift as the float ub with bits 0x4B400000 + u
      // (1.5·2^23 + u).  t = RD(ub·cs + (1.5·2^23 - 1.5·2^23·cs)), with
      // cs = c17/2^17 and both terms exact (1.5·2^23·cs = 96·c17), is
      // RD(u·cs + 1.5·2^23) = 1.5·2^23 + ⌊u/s⌋ (the grid there is the
      // integers, and u·c17/2^17 is within u/2^17 < 1/s of u/s);
      // d1 = t - (1.5·2^23 + h1), d0 = (u - h0 - s·h1) - s·d1.  Every value
      // is an integer below 2^24, exact in FP32, and the FP32 pipes take
      // this work off the integer multiply pipe the residue sums load.
      const float ub = __int_as_float(static_cast<int>(static_cast<uint32_t>(off) + (0x4B400000u + kShift)));
      const float uh = ub - static_cast<float>(12582912 + mc.sq_h0 + mc.s * mc.sq_h1);
      const float t = __fmaf_rd(ub, static_cast<float>(mc.sq_c17) * (1.0f / 131072.0f),
                                static_cast<float>(12582912 - 96 * mc.sq_c17));
      f1[e] = t - static_cast<float>(12582912 + mc.sq_h1);
      f0[e] = __fmaf_rn(-static_cast<float>(mc.s), f1[e], uh);
    }
  }
  uint8_t* pdst = dst + (mc.plane_off - PBASE) * STRIDE;
  *reinterpret_cast<uint2*>(pdst) = make_uint2(__byte_perm(e4m3x2(f0[0], f0[1]), e4m3x2(f0[2], f0[3]), 0x5410),
                                               __byte_perm(e4m3x2(f0[4], f0[5]), e4m3x2(f0[6], f0[7]), 0x5410));
  *reinterpret_cast<uint2*>(pdst + STRIDE) =
      make_uint2(__byte_perm(e4m3x2(f1[0], f1[1]), e4m3x2(f1[2], f1[3]), 0x5410),
                 __byte_perm(e4m3x2(f1[4], f1[5]), e4m3x2(f1[6], f1[7]), 0x5410));
}

template <int I, int STRIDE = kPlaneBlock, int PBASE = 0>
__device__ __forceinline__ void planes_one(const Limbs& L, const uint32_t* table, uint8_t* dst) {
  constexpr ModConst mc = mod_const(I);
  if constexpr (mc.s != 0) {
    square_digits<I, STRIDE, PBASE>(L, dst);
    return;
  }
  const uint32_t* centre = table + mc.table_off + mc.m;
  uint32_t w[kElems];
#pragma unroll
  for (int e = 0; e < kElems; ++e) {
    const uint32_t Y = L.w0[e] + L.w1[e] * static_cast<uint32_t>(mc.c1) +
                       static_cast<uint32_t>(L.w2[e]) * static_cast<uint32_t>(mc.c2);
    const uint32_t q = __umulhi(Y, mc.magic);
    const int off = static_cast<int>(Y - q * static_cast<uint32_t>(mc.m));  // in [-m, m)
    w[e] = centre[off];  // packed E4M3 planes of centred(Ã mod m)
  }
  uint8_t* pdst = dst + (mc.plane_off - PBASE) * STRIDE;
  uint32_t lo[3], hi[3];
  transpose3(w[0], w[1], w[2], w[3], lo[0], lo[1], lo[2]);
  transpose3(w[4], w[5], w[6], w[7], hi[0], hi[1], hi[2]);
#pragma unroll
  for (int p = 0; p < 3; ++p) *reinterpret_cast<uint2*>(pdst + p * STRIDE) = make_uint2(lo[p], hi[p]);
}

template <int... Is>
__device__ __forceinline__ void planes_all(std::integer_sequence<int, Is...>, const Limbs& L, const uint32_t* table,
                                           uint8_t* dst) {
  (planes_one<Is>(L, table, dst), ...);
}

// MODE 0: magnitude plane (1 plane); MODE 1: residue digit planes for the
// first R moduli (R is a template parameter so the modulus loop unrolls and
// every per-modulus constant and plane offset is known at compile time).
template <int MODE, int R>
__global__ void __launch_bounds__(TileShape<MODE>::kThreads, TileShape<MODE>::kBlocksPerSm) planes_kernel(OperandView X0, OperandView X1, int blocks0, int64_t k,
                                                             int64_t k_pad, int clamp_c, int rn,
                                                             const __grid_constant__ Oz2Moduli mods) {
  extern __shared__ uint32_t table[];
  const bool second = static_cast<int>(blockIdx.x) >= blocks0;
  const OperandView X = second ? X1 : X0;
  const int bid = second ? blockIdx.x - blocks0 : blockIdx.x;
  const int nblocks = second ? gridDim.x - blocks0 : blocks0;
  if (MODE == 1) {
    for (int t = threadIdx.x; t < mods.table_entries; t += blockDim.x) table[t] = X.table[t];
    __syncthreads();
  }
  using TS = TileShape<MODE>;
  const int64_t rows_out = rows_stored<MODE>(X.rows);
  const int64_t row_tiles = (rows_out + TS::kRows - 1) / TS::kRows;
  const int64_t ntiles = row_tiles * (k_pad / TS::kSeg);
  const int part = threadIdx.x & (TS::kThreadsPerRow - 1);
  const int rloc = threadIdx.x / TS::kThreadsPerRow;

  for (int64_t tile = bid; tile < ntiles; tile += nblocks) {
    const int64_t kt = tile / row_tiles;  // consecutive blocks share a k-slice of many rows
    const int64_t row = (tile - kt * row_tiles) * TS::kRows + rloc;
    if (row >= rows_out) continue;
    const int64_t l0 = kt * TS::kSeg + part * kElems;
    const bool pad = row >= X.rows;  // pad rows of the last block: zero digits
    double x[kElems];
    if (pad) {
#pragma unroll
      for (int e = 0; e < kElems; ++e) x[e] = 0.0;
    } else {
      load8(X, row, l0, k, x);  // entries of rows zeroed by the flags are replaced below
    }
    const bool zero_row = pad || (X.flag[row] & 2) != 0;
    const int ex = pad ? 0 : X.exps[row];
    // Magnitude plane: row-major rows × k_pad.  Digit planes: 128 × 128-byte
    // blocks, those of one (row block, k-block) consecutive.
    uint8_t* dst =
        MODE == 0 ? X.out + static_cast<size_t>(row) * k_pad + l0
                  : X.out + ((static_cast<size_t>(row / kPlaneRows) * (k_pad / kPlaneLine) + l0 / kPlaneLine) *
                                 num_planes(R) * kPlaneBlock +
                             (row % kPlaneRows) * kPlaneLine + l0 % kPlaneLine);
    const bool fast_tz = MODE == 1 && !rn && ex <= kTzFastMaxD;
    if (zero_row && !fast_tz) {  // the fast truncating path zeroes through its scale
#pragma unroll
      for (int e = 0; e < kElems; ++e) x[e] = 0.0;
    }

    if (MODE == 0) {
      uint32_t code[kElems];
#pragma unroll
      for (int e = 0; e < kElems; ++e) code[e] = magnitude_code(x[e], ex, clamp_c);
      *reinterpret_cast<uint2*>(dst) = make_uint2(code[0] | (code[1] << 8) | (code[2] << 16) | (code[3] << 24),
                                                  code[4] | (code[5] << 8) | (code[6] << 16) | (code[7] << 24));
    } else {
      // Quantise (Eq. scale) and split Ã, a 64-bit two's complement word,
      // into 21-bit limbs.
      Limbs L;
      if (fast_tz) {
        const int d = zero_row ? -4096 : ex;
#pragma unroll
        for (int e = 0; e < kElems; ++e) quantise_tz_limbs(x[e], d, L, e);
      } else {
#pragma unroll
        for (int e = 0; e < kElems; ++e) {
          const Split sp = split_double(x[e]);
          const unsigned long long a = quantise_abs(sp, ex, rn != 0);
          const unsigned long long t = sp.neg ? 0ull - a : a;
          set_limbs(L, e, static_cast<uint32_t>(t), static_cast<int>(t >> 32));
        }
      }
      planes_all(std::make_integer_sequence<int, R>{}, L, table, dst);
    }
  }
}


// ---------------------------------------------------------------------------
// On-the-fly residues for a skinny C (n ≤ 32): the residue GEMM with A's
// digit planes formed in shared memory straight from A (the paper's plane
// storage mode F, §"plane-storage modes" and Appendix E), so they are never
// written to HBM and read back: for n ≤ 32 every element of A feeds one tile
// column, and storing its 30 plane bytes (r = 12) would cost far more
// traffic than the 8 bytes of A the conversion reads.
//
// A CTA takes 128 rows of A and every column of C.  Each 32-entry k-chunk
// (one MMA K-step) is converted once: 512 threads, four per row, quantise
// 8 entries each (Eq. scale) and split them into limbs; the moduli then go in
// groups of up to six, each group's digit planes written by the same
// per-modulus code as the deconstruction into one of two shared-memory
// buffers (with the group's B plane tiles, copied from B's deconstruction),
// so that the tensor core consumes one group while the threads convert the
// next.  The A and B tiles are K-major without swizzle: 8-row × 16-byte core
// matrices, the two 16-byte halves of a 32-byte row 2 KiB (A) or 16·N bytes
// (B) apart.
//
// Modulus blocking (Eq. nblk, Eq. blkcost): the accumulator pairs of a
// modulus take 2·N TMEM columns, so a pass holds 256/N moduli (every modulus
// for N = 16, eight for N = 32); each pass sweeps all of k and reads A again
// (the cost Eq. blkcost prices), with its accumulators resident.  Every
// 4096 k-entries (Eq. accum-exact for the merged accumulator) the threads
// reduce the accumulators mod m and write the residue back for the next
// K-slab to accumulate on (as the residue GEMM does); after the last they
// store the centred residues C^(i).
// ---------------------------------------------------------------------------
constexpr int kMfKc = 32;                              // k-entries per chunk (one MMA K-step)
constexpr int kMfThreads = 512;                        // 128 rows × 4 threads (8 entries each)
constexpr int kMfAPlane = kRows * kMfKc;               // 4 KiB: an A plane tile of one chunk
constexpr int kMfGroup = 6;                            // moduli per shared-memory group
constexpr int kMfGroupPlanes = 3 * kMfGroup;           // planes a group holds at most
constexpr int kMfSlabChunks = kKSlabMerged / kMfKc;    // chunks per K-slab
constexpr long long kMfWaitLimit = 2000000000LL;       // ≈1 s at 2 GHz

template <int NT>
struct ModeFShape {
  static constexpr int kBPlane = NT * kMfKc;                          // a B plane tile of one chunk
  static constexpr int kBOff = kMfGroupPlanes * kMfAPlane;            // B tiles after the A tiles
  static constexpr int kBuf = kBOff + kMfGroupPlanes * kBPlane;       // one group buffer
  static constexpr int kPassModuli = 256 / NT;                        // moduli a TMEM pass holds
  static constexpr int kCols = NT / 4;                                // epilogue columns per thread
};

struct ModeFArgs {
  const double* A;
  int64_t lda, m, n, k, k_pad;
  const int32_t* d;
  const uint8_t* row_flag;
  const uint8_t* planes_b;
  int16_t* res;
  int64_t ldr;
  int rn;
  Oz2Device* dev;
};

struct ModeFState {
  uint8_t* buf[2];
  uint32_t bar[2];   // completions of the MMAs that read each buffer
  uint32_t tmem;
  uint32_t item;     // group-chunks issued so far
  bool ok;
};

// Digit planes of moduli [G0, G1) for this thread's 8 entries, into `slot`
// (the thread's 8-byte place in plane 0 of the group buffer).
template <int G0, int... Js>
__device__ __forceinline__ void modef_convert(std::integer_sequence<int, Js...>, const Limbs& L,
                                              const uint32_t* table, uint8_t* slot) {
  constexpr int kBase = mod_const(G0).plane_off;
  (planes_one<G0 + Js, kMfAPlane, kBase>(L, table, slot), ...);
}

// One group of moduli [G0, G1) for chunk c: its planes into the next buffer,
// its B tiles beside them, then its MMAs into the pass's accumulators
// (moduli from P0 on).
template <int R, int NT, int P0, int G0, int G1>
__device__ __forceinline__ void modef_group(ModeFState& st, const ModeFArgs& a, const Oz2Moduli& mods,
                                            const uint32_t* table, int64_t c, const Limbs& L) {
  using S = ModeFShape<NT>;
  constexpr int kBase = mod_const(G0).plane_off;
  constexpr int kPlanes = num_planes(G1) - kBase;
  const int tid = threadIdx.x;
  const uint32_t bi = st.item & 1;
  uint8_t* buf = st.buf[bi];
  // The buffer is free once the MMAs of two group-chunks ago completed.
  if (st.item >= 2 && !mbar_wait_bounded(st.bar[bi], ((st.item >> 1) & 1) ^ 1, kMfWaitLimit)) st.ok = false;
  const int row = tid >> 2, part = tid & 3;
  modef_convert<G0>(std::make_integer_sequence<int, G1 - G0>{}, L, table,
                    buf + (part >> 1) * (kMfAPlane / 2) + row * 16 + (part & 1) * 8);
  // B tiles: rows 0..NT-1 of B's planes for this chunk (all in B's first
  // 128-row block; rows past n are the storage's zero pad rows), two 16-byte
  // halves each.
  for (int t = tid; t < kPlanes * NT * 2; t += kMfThreads) {
    const int j = t / (NT * 2), rr = (t >> 1) % NT, h = t & 1;
    const uint8_t* src = a.planes_b + (c * kMfKc / kPlaneLine) * mods.nplanes * kPlaneBlock +
                         static_cast<int64_t>(kBase + j) * kPlaneBlock + rr * kPlaneLine + (c * kMfKc) % kPlaneLine +
                         16 * h;
    *reinterpret_cast<uint4*>(buf + S::kBOff + j * S::kBPlane + h * (NT * 16) + rr * 16) =
        __ldg(reinterpret_cast<const uint4*>(src));
  }
  fence_proxy_async_smem();  // the tensor core reads what the threads wrote
  // A wait that expired in any thread stops the whole block here.
  if (__syncthreads_or(!st.ok)) {
    st.ok = false;
    return;
  }
  if (tid == 0) {
    tc_fence_after();
    constexpr uint32_t idesc = idesc_f8_f32(kRows, NT);
    const uint32_t a0 = smem_u32(buf), b0 = smem_u32(buf + S::kBOff);
    const uint32_t first = (c % kMfSlabChunks == 0 && c < kMfSlabChunks) ? 0u : 1u;
#pragma unroll
    for (int i = G0; i < G1; ++i) {
      const int j = mods.plane_off[i] - kBase;
      const uint32_t acc0 = st.tmem + static_cast<uint32_t>((i - P0) * 2 * NT), acc1 = acc0 + NT;
      auto ad = [&](int p) { return smem_desc_plain(a0 + (j + p) * kMfAPlane, kMfAPlane / 2, 128); };
      auto bd = [&](int p) { return smem_desc_plain(b0 + (j + p) * S::kBPlane, NT * 16, 128); };
      if (mods.sq_base[i]) {
        mma_f8(acc0, ad(0), bd(0), idesc, first);  // d0·e0
        mma_f8(acc1, ad(1), bd(0), idesc, first);  // d1·e0
        mma_f8(acc1, ad(0), bd(1), idesc, 1u);     // + d0·e1
      } else {
        mma_f8(acc0, ad(0), bd(0), idesc, first);  // Σ·Σ
        mma_f8(acc1, ad(1), bd(1), idesc, first);  // d0·e0
        mma_f8(acc1, ad(2), bd(2), idesc, 1u);     // + (-16 d1)·e1
      }
    }
    mma_commit(st.bar[bi]);
  }
  ++st.item;
}

template <int R, int NT, int P0, int P1, int G0>
__device__ __forceinline__ void modef_groups(ModeFState& st, const ModeFArgs& a, const Oz2Moduli& mods,
                                             const uint32_t* table, int64_t c, const Limbs& L) {
  if constexpr (G0 < P1) {
    constexpr int G1 = G0 + kMfGroup < P1 ? G0 + kMfGroup : P1;
    modef_group<R, NT, P0, G0, G1>(st, a, mods, table, c, L);
    if (st.ok) modef_groups<R, NT, P0, P1, G1>(st, a, mods, table, c, L);
  }
}

// The accumulators of moduli [P0, P1) after a K-slab: each thread reduces its
// row's NT/4 columns of every modulus to the centred residue, and either
// writes it back for the next slab (acc0 = r and acc1 = 0 for a square
// modulus, v = acc0 + s·acc1; acc0 = acc1 = r otherwise, 16r - 15r = r) or
// stores it as C^(i).
template <int NT, int P0, int P1>
__device__ __forceinline__ void modef_epilogue(ModeFState& st, const ModeFArgs& a, const Oz2Moduli& mods,
                                               int64_t row0, bool last) {
  using S = ModeFShape<NT>;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int q = warp & 3, cg = warp >> 2;
  const int64_t row = row0 + 32 * q + lane;
  const uint32_t lane_addr = st.tmem + (static_cast<uint32_t>(32 * q) << 16) + static_cast<uint32_t>(S::kCols * cg);
  for (int i = P0; i < P1; ++i) {
    const bool square = mods.sq_base[i] != 0;
    const float mf = static_cast<float>(mods.m[i]), inv = 1.f / mf, sb = static_cast<float>(mods.sq_base[i]);
    const float hi = static_cast<float>(mods.m[i] - 1 - mods.m[i] / 2);
#pragma unroll
    for (int c4 = 0; c4 < S::kCols; c4 += 4) {
      const uint32_t at = lane_addr + static_cast<uint32_t>((i - P0) * 2 * NT + c4);
      uint32_t v0[4], v1[4];
      tmem_ld4(at, v0);
      tmem_ld4(at + NT, v1);
      tmem_ld_wait();
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float r = combine_residue(__uint_as_float(v0[j]), __uint_as_float(v1[j]), square, sb, mf, inv, hi, 0.f);
        v0[j] = __float_as_uint(r);
        v1[j] = square ? 0u : v0[j];
        const int64_t col = S::kCols * cg + c4 + j;
        if (last && row < a.m && col < a.n)
          a.res[(static_cast<size_t>(i) * a.n + col) * a.ldr + row] = static_cast<int16_t>(as_i16_bits(r));
      }
      if (!last) {
        tmem_st4(at, v0);
        tmem_st4(at + NT, v1);
      }
    }
  }
  if (!last) tmem_st_wait();
}

// One pass over moduli [P0, P1) for the 128 rows from row0: every chunk of k,
// converted once and fed group by group, with a reduction at each K-slab end.
template <int R, int NT, int P0, int P1>
__device__ __forceinline__ void modef_pass(ModeFState& st, const ModeFArgs& a, const Oz2Moduli& mods,
                                           const uint32_t* table, int64_t row0) {
  const int tid = threadIdx.x;
  const int64_t row = row0 + (tid >> 2);
  const int part = tid & 3;
  const bool pad = row >= a.m;
  const bool zero_row = pad || (a.row_flag[row] & 2) != 0;
  const int ex = pad ? 0 : a.d[row];
  const bool fast_tz = !a.rn && ex <= kTzFastMaxD;
  const int64_t nchunks = a.k_pad / kMfKc;
  // This thread's 8 entries of chunk c (zero past k and on pad rows).
  auto load = [&](int64_t c, double (&x)[kElems]) {
    const int64_t l0 = c * kMfKc + part * kElems;
    const double* p = a.A + row + l0 * a.lda;
#pragma unroll
    for (int e = 0; e < kElems; ++e) x[e] = !pad && l0 + e < a.k ? __ldg(p + e * a.lda) : 0.0;
  };
  double xn[kElems];
  load(0, xn);
  for (int64_t c = 0; c < nchunks && st.ok; ++c) {
    double x[kElems];
#pragma unroll
    for (int e = 0; e < kElems; ++e) x[e] = xn[e];
    if (c + 1 < nchunks) load(c + 1, xn);  // in flight while this chunk is converted
    if (zero_row && !fast_tz) {
#pragma unroll
      for (int e = 0; e < kElems; ++e) x[e] = 0.0;
    }
    Limbs L;
    if (fast_tz) {
      const int dd = zero_row ? -4096 : ex;
#pragma unroll
      for (int e = 0; e < kElems; ++e) quantise_tz_limbs(x[e], dd, L, e);
    } else {
#pragma unroll
      for (int e = 0; e < kElems; ++e) {
        const Split sp = split_double(x[e]);
        const unsigned long long aa = quantise_abs(sp, ex, a.rn != 0);
        const unsigned long long t = sp.neg ? 0ull - aa : aa;
        set_limbs(L, e, static_cast<uint32_t>(t), static_cast<int>(t >> 32));
      }
    }
    modef_groups<R, NT, P0, P1, P0>(st, a, mods, table, c, L);
    if (!st.ok) break;
    const bool slab_end = (c + 1) % kMfSlabChunks == 0 || c + 1 == nchunks;
    if (slab_end) {
      // Every MMA so far retired (the last commit covers the earlier ones).
      const uint32_t li = st.item - 1;
      if (!mbar_wait_bounded(st.bar[li & 1], (li >> 1) & 1, kMfWaitLimit)) st.ok = false;
      tc_fence_after();
      modef_epilogue<NT, P0, P1>(st, a, mods, row0, c + 1 == nchunks);
      tc_fence_before();
      // The next MMAs write these accumulators; an expired wait stops the block.
      if (__syncthreads_or(!st.ok)) st.ok = false;
    }
  }
}

template <int R, int NT, int P0>
__device__ __forceinline__ void modef_passes(ModeFState& st, const ModeFArgs& a, const Oz2Moduli& mods,
                                             const uint32_t* table, int64_t row0) {
  if constexpr (P0 < R) {
    constexpr int P1 = P0 + ModeFShape<NT>::kPassModuli < R ? P0 + ModeFShape<NT>::kPassModuli : R;
    modef_pass<R, NT, P0, P1>(st, a, mods, table, row0);
    modef_passes<R, NT, P1>(st, a, mods, table, row0);
  }
}

template <int R, int NT>
__global__ void __launch_bounds__(kMfThreads, 1) modef_kernel(const __grid_constant__ Oz2Moduli mods, ModeFArgs a,
                                                              const uint32_t* __restrict__ table_a) {
  using S = ModeFShape<NT>;
  extern __shared__ __align__(1024) uint8_t mf_smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(mf_smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + 2 * S::kBuf);
  uint32_t* table = reinterpret_cast<uint32_t*>(sm + 2 * S::kBuf + 64);
  __shared__ uint32_t tmem_base_s;
  const int tid = threadIdx.x, warp = tid >> 5;
  for (int t = tid; t < mods.table_entries; t += kMfThreads) table[t] = table_a[t];
  if (tid == 0) {
    mbar_init(smem_u32(bars), 1);
    mbar_init(smem_u32(bars + 1), 1);
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(&tmem_base_s), 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  ModeFState st{{sm, sm + S::kBuf}, {smem_u32(bars), smem_u32(bars + 1)}, tmem_base_s, 0u, true};
  const int64_t nrb = (a.m + kRows - 1) / kRows;
  for (int64_t rb = blockIdx.x; rb < nrb && st.ok; rb += gridDim.x) modef_passes<R, NT, 0>(st, a, mods, table, rb * kRows);
  // Every MMA retired before the tensor memory goes away.
  if (st.item > 0) {
    const uint32_t li = st.item - 1;
    mbar_wait_bounded(st.bar[li & 1], (li >> 1) & 1, kMfWaitLimit);
  }
  if (!st.ok && tid == 0) {
    a.dev->status = kStatusTimeout;
    a.dev->timeout_site = 10;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0) tmem_dealloc(st.tmem, 512);
}

bool modef_applies(int64_t m, int64_t n, int64_t k_pad) { return n <= kModeFMaxN && m >= kRows && k_pad >= 1024; }

template <int NT>
static size_t modef_smem(const Oz2Moduli& mods) {
  return 1024 + 2 * ModeFShape<NT>::kBuf + 64 + sizeof(uint32_t) * static_cast<size_t>(mods.table_entries);
}

template <int R, int NT>
static cudaError_t launch_modef_rn(const Oz2Moduli& mods, const ModeFArgs& a, const uint32_t* table_a,
                                   cudaStream_t st) {
  const size_t smem = modef_smem<NT>(mods);
  cudaError_t err =
      cudaFuncSetAttribute(modef_kernel<R, NT>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (err != cudaSuccess) return err;
  const int64_t grid = std::min<int64_t>(num_sms(), (a.m + kRows - 1) / kRows);
  count_launch();
  modef_kernel<R, NT><<<static_cast<unsigned>(grid), kMfThreads, smem, st>>>(mods, a, table_a);
  return cudaGetLastError();
}

template <int R>
static cudaError_t launch_modef_r(const Oz2Moduli& mods, const ModeFArgs& a, const uint32_t* table_a,
                                  cudaStream_t st) {
  return a.n <= 16 ? launch_modef_rn<R, 16>(mods, a, table_a, st) : launch_modef_rn<R, 32>(mods, a, table_a, st);
}

cudaError_t launch_modef(int64_t m, int64_t n, int64_t k, const Oz2Moduli& mods, const uint32_t* table_a,
                         const double* A, int64_t lda, const int32_t* d, const uint8_t* row_flag, int quant,
                         const uint8_t* planes_b, int16_t* residues, int64_t ldr, Oz2Device* dev, cudaStream_t st) {
  if (m == 0 || n == 0) return cudaSuccess;
  const int64_t k_pad = (k + kKPad - 1) / kKPad * kKPad;
  if (!modef_applies(m, n, k_pad)) return cudaErrorInvalidValue;
  const ModeFArgs a{A, lda, m, n, k, k_pad, d, row_flag, planes_b, residues, ldr, quant == OZ2_QUANT_RN, dev};
  switch (mods.r) {
#define OZ2_MF_CASE(R) \
  case R:              \
    return launch_modef_r<R>(mods, a, table_a, st);
    OZ2_MF_CASE(1) OZ2_MF_CASE(2) OZ2_MF_CASE(3) OZ2_MF_CASE(4) OZ2_MF_CASE(5) OZ2_MF_CASE(6)
    OZ2_MF_CASE(7) OZ2_MF_CASE(8) OZ2_MF_CASE(9) OZ2_MF_CASE(10) OZ2_MF_CASE(11) OZ2_MF_CASE(12)
    OZ2_MF_CASE(13) OZ2_MF_CASE(14) OZ2_MF_CASE(15) OZ2_MF_CASE(16)
#undef OZ2_MF_CASE
    default:
      return cudaErrorInvalidValue;
  }
}

template <int MODE>
static int64_t tiles_of(int64_t rows, int64_t k_pad) {
  using TS = TileShape<MODE>;
  return ((rows_stored<MODE>(rows) + TS::kRows - 1) / TS::kRows) * (k_pad / TS::kSeg);
}

// Split a grid of about `blocks_per_sm` × SMs blocks between the two operands
// in proportion to their tiles.
static void split_grid(int64_t t0, int64_t t1, int blocks_per_sm, int* g0, int* g1) {
  const int64_t cap = static_cast<int64_t>(num_sms()) * blocks_per_sm;
  const int64_t tot = t0 + t1;
  int64_t b0 = t0 ? std::max<int64_t>(1, std::min<int64_t>(t0, cap * t0 / std::max<int64_t>(tot, 1))) : 0;
  int64_t b1 = t1 ? std::max<int64_t>(1, std::min<int64_t>(t1, cap - b0)) : 0;
  *g0 = static_cast<int>(b0);
  *g1 = static_cast<int>(b1);
}

static int vec_ok(const double* base, int64_t row_stride, int64_t k_stride) {
  return k_stride == 1 && (row_stride % 2 == 0) && (reinterpret_cast<uintptr_t>(base) % 16 == 0);
}

cudaError_t launch_magnitude_planes(int64_t m, int64_t n, int64_t k, const double* A,
                                    int64_t lda, const double* B, int64_t ldb, const int32_t* ra,
                                    const int32_t* cb, const uint8_t* row_flag,
                                    const uint8_t* col_flag, uint8_t* mag_a, uint8_t* mag_b,
                                    cudaStream_t st) {
  const int64_t k_pad = (k + kKPad - 1) / kKPad * kKPad;
  int lk = k <= 1 ? 0 : 64 - __builtin_clzll(static_cast<unsigned long long>(k - 1));
  int c = (24 - lk) / 2;
  c = c < 0 ? 0 : (c > kMagClampMax ? kMagClampMax : c);
  Oz2Moduli dummy{};
  OperandView va{A, 1, lda, m, ra, row_flag, mag_a, nullptr, 0};
  OperandView vb{B, ldb, 1, n, cb, col_flag, mag_b, nullptr, vec_ok(B, ldb, 1)};
  int g0, g1;
  split_grid(m ? tiles_of<0>(m, k_pad) : 0, n ? tiles_of<0>(n, k_pad) : 0, TileShape<0>::kBlocksPerSm, &g0, &g1);
  if (g0 + g1 == 0) return cudaSuccess;
  if (g0 == 0) va = vb;
  count_launch();
  planes_kernel<0, 0><<<g0 + g1, TileShape<0>::kThreads, 0, st>>>(va, vb, g0, k, k_pad, c, 0, dummy);
  return cudaGetLastError();
}

cudaError_t launch_deconstruct(int64_t m, int64_t n, int64_t k, const Oz2Moduli& mods,
                               const uint32_t* table_a, const uint32_t* table_b, const double* A, int64_t lda,
                               const double* B, int64_t ldb, const int32_t* d, const int32_t* e,
                               const uint8_t* row_flag, const uint8_t* col_flag, int quant,
                               uint8_t* planes_a, uint8_t* planes_b, cudaStream_t st) {
  const int64_t k_pad = (k + kKPad - 1) / kKPad * kKPad;
  const size_t smem = sizeof(uint32_t) * mods.table_entries;
  const int rn = quant == OZ2_QUANT_RN;
  OperandView va{A, 1, lda, m, d, row_flag, planes_a, table_a, 0};
  OperandView vb{B, ldb, 1, n, e, col_flag, planes_b, table_b, vec_ok(B, ldb, 1)};
  int g0, g1;
  split_grid(m ? tiles_of<1>(m, k_pad) : 0, n ? tiles_of<1>(n, k_pad) : 0, TileShape<1>::kBlocksPerSm, &g0, &g1);
  if (g0 + g1 == 0) return cudaSuccess;
  if (g0 == 0) va = vb;
  cudaError_t err = cudaSuccess;
  count_launch();
  switch (mods.r) {
#define OZ2_DEC_CASE(R)                                                                                     \
  case R:                                                                                                   \
    err = cudaFuncSetAttribute(planes_kernel<1, R>, cudaFuncAttributeMaxDynamicSharedMemorySize,            \
                               static_cast<int>(smem));                                                     \
    if (err == cudaSuccess)                                                                                 \
      planes_kernel<1, R><<<g0 + g1, TileShape<1>::kThreads, smem, st>>>(va, vb, g0, k, k_pad, 0, rn, mods); \
    break;
    OZ2_DEC_CASE(1) OZ2_DEC_CASE(2) OZ2_DEC_CASE(3) OZ2_DEC_CASE(4) OZ2_DEC_CASE(5) OZ2_DEC_CASE(6)
    OZ2_DEC_CASE(7) OZ2_DEC_CASE(8) OZ2_DEC_CASE(9) OZ2_DEC_CASE(10) OZ2_DEC_CASE(11) OZ2_DEC_CASE(12)
    OZ2_DEC_CASE(13) OZ2_DEC_CASE(14) OZ2_DEC_CASE(15) OZ2_DEC_CASE(16)
#undef OZ2_DEC_CASE
    default:
      return cudaErrorInvalidValue;
  }
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

}  // namespace oz2
