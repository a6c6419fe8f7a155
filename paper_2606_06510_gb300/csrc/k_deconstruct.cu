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

#include "oz2_common.cuh"

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

// Truncating quantisation (Eq. scale, TZ) of one entry into the limbs the
// residue sums take: Ã = trunc(x·2^d) as a 64-bit two's complement word,
// for rows with d ≤ kTzFastMaxD, split into
// b = 4·(bits 0-15 + kDecBias), bits 16-31, bits 32-47 and the signed bits
// 48-63.  With x = ±M·2^(sh - d), M < 2^53, Ã = ±⌊M·2^10 / 2^(10 - sh)⌋: the
// significand is shifted up by 10 (below 2^63) and then right by r = 10 - sh
// with clamping funnel shifts, so zeros, subnormals and entries that shift
// out entirely need no branch.  That needs sh ≤ 9: a normal x has M ≥ 2^52
// and |Ã| < 2^62, and a subnormal one has sh = d - 1074 ≤ 9 for
// d ≤ kTzFastMaxD (rows with a larger scale, whose largest entry is itself
// subnormal, take the general path).  d = -4096 gives Ã = 0 for any x.
constexpr int kTzFastMaxD = 1083;
__device__ __forceinline__ void quantise_tz_limbs(double x, int d, uint32_t& b, uint32_t& u1, uint32_t& u2,
                                                  int& u3) {
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
  const uint32_t tl = static_cast<uint32_t>(t);
  const int th = static_cast<int>(t >> 32);
  b = ((tl << 2) & 0x3FFFCu) | (4u * kDecBias);
  u1 = tl >> 16;
  u2 = static_cast<uint32_t>(th) & 0xFFFFu;
  u3 = th >> 16;
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

// Gather byte `b` of four 32-bit words into one word (byte 0 from w0 ...).
__device__ __forceinline__ uint32_t gather_byte(uint32_t w0, uint32_t w1, uint32_t w2, uint32_t w3,
                                                int b) {
  uint32_t sel = static_cast<uint32_t>(b) | (static_cast<uint32_t>(b + 4) << 4);
  uint32_t lo = __byte_perm(w0, w1, sel);       // bytes: w0.b, w1.b
  uint32_t hi = __byte_perm(w2, w3, sel);       // bytes: w2.b, w3.b
  return __byte_perm(lo, hi, 0x5410);
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
// Ã = u0 + u1·2^16 + u2·2^32 + u3·2^48 with u3 signed (|Ã| < 2^62, so
// |u3| ≤ 2^14), and b = 4·(u0 + kDecBias).  Then
//   Y = b + 4·(u1·(2^16 mod m) + u2·(2^32 mod m) + u3·(2^48 mod m))
// is 4·y with y ≡ Ã + kDecBias (mod m) and 2^24 < y < 2^28 (the bias
// outweighs the most negative u3 term).  With magic = ⌈2^30/m⌉,
// q = ⌊Y·magic/2^32⌋ = ⌊y/m + y·(magic·m - 2^30)/(m·2^30)⌋ is ⌊y/m⌋ or one
// more, since the second term is below y/2^30 < 1; so Y - 4qm = 4(y - qm) is
// the byte offset of the entry for y mod m in a table whose 2m entries
// start m entries before it.  The table is rotated by kDecBias.
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
// d0 = (u mod s) - h0 and d1 = ⌊u/s⌋ - h1.  u = ((y + E) mod m) + h0 + s·h1 -
// ⌊m/2⌋, since c = ((x + ⌊m/2⌋) mod m) - ⌊m/2⌋ for x = Ã mod m = (y - B)
// mod m.  (y + E) mod m comes from the same shifted magic quotient as the
// table index, corrected once.
template <int I>
__device__ __forceinline__ void square_digits(const uint32_t (&b)[kElems], const uint32_t (&u1)[kElems],
                                              const uint32_t (&u2)[kElems], const int (&u3)[kElems],
                                              uint8_t* dst) {
  constexpr ModConst mc = mod_const(I);
  constexpr int kShift = mc.sq_h0 + mc.s * mc.sq_h1 - mc.m / 2;  // u - (y + E) mod m, ≥ 0
  float f0[kElems], f1[kElems];
#pragma unroll
  for (int e = 0; e < kElems; ++e) {
    const uint32_t Y = b[e] + 4 * mc.sq_e + u1[e] * mc.limb1 + u2[e] * mc.limb2 +
                       static_cast<uint32_t>(u3[e]) * mc.limb3;
    const uint32_t q = __umulhi(Y, mc.magic);
    int off = static_cast<int>(Y - q * static_cast<uint32_t>(4 * mc.m));  // 4·((y + E) mod m) or that - 4m
    off += off < 0 ? 4 * mc.m : 0;
    const uint32_t u = (static_cast<uint32_t>(off) >> 2) + kShift;
    const uint32_t a1 = mc.s == 32 ? u >> 5 : __umulhi(u, mc.sq_magic);
    const uint32_t a0 = u - a1 * static_cast<uint32_t>(mc.s);
    f0[e] = small_int_float(a0 + (0x4B400000u - mc.sq_h0));
    f1[e] = small_int_float(a1 + (0x4B400000u - mc.sq_h1));
  }
  uint8_t* pdst = dst + mc.plane_off * kPlaneBlock;
  *reinterpret_cast<uint2*>(pdst) = make_uint2(__byte_perm(e4m3x2(f0[0], f0[1]), e4m3x2(f0[2], f0[3]), 0x5410),
                                               __byte_perm(e4m3x2(f0[4], f0[5]), e4m3x2(f0[6], f0[7]), 0x5410));
  *reinterpret_cast<uint2*>(pdst + kPlaneBlock) =
      make_uint2(__byte_perm(e4m3x2(f1[0], f1[1]), e4m3x2(f1[2], f1[3]), 0x5410),
                 __byte_perm(e4m3x2(f1[4], f1[5]), e4m3x2(f1[6], f1[7]), 0x5410));
}

template <int I>
__device__ __forceinline__ void planes_one(const uint32_t (&b)[kElems], const uint32_t (&u1)[kElems],
                                           const uint32_t (&u2)[kElems], const int (&u3)[kElems],
                                           const uint32_t* table, uint8_t* dst) {
  constexpr ModConst mc = mod_const(I);
  if constexpr (mc.s != 0) {
    square_digits<I>(b, u1, u2, u3, dst);
    return;
  }
  const char* centre = reinterpret_cast<const char*>(table + mc.table_off + mc.m);
  uint32_t w[kElems];
#pragma unroll
  for (int e = 0; e < kElems; ++e) {
    const uint32_t Y = b[e] + u1[e] * mc.limb1 + u2[e] * mc.limb2 + static_cast<uint32_t>(u3[e]) * mc.limb3;
    const uint32_t q = __umulhi(Y, mc.magic);
    const int off = static_cast<int>(Y - q * static_cast<uint32_t>(4 * mc.m));  // in [-4m, 4m)
    w[e] = *reinterpret_cast<const uint32_t*>(centre + off);  // packed E4M3 planes of centred(Ã mod m)
  }
  uint8_t* pdst = dst + mc.plane_off * kPlaneBlock;
#pragma unroll
  for (int p = 0; p < (mc.s ? 2 : 3); ++p)
    *reinterpret_cast<uint2*>(pdst + p * kPlaneBlock) =
        make_uint2(gather_byte(w[0], w[1], w[2], w[3], p), gather_byte(w[4], w[5], w[6], w[7], p));
}

template <int... Is>
__device__ __forceinline__ void planes_all(std::integer_sequence<int, Is...>, const uint32_t (&b)[kElems],
                                           const uint32_t (&u1)[kElems], const uint32_t (&u2)[kElems],
                                           const int (&u3)[kElems], const uint32_t* table, uint8_t* dst) {
  (planes_one<Is>(b, u1, u2, u3, table, dst), ...);
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
      // into three unsigned 16-bit limbs and a signed top limb.
      uint32_t b[kElems], u1[kElems], u2[kElems];
      int u3[kElems];
      if (fast_tz) {
        const int d = zero_row ? -4096 : ex;
#pragma unroll
        for (int e = 0; e < kElems; ++e) quantise_tz_limbs(x[e], d, b[e], u1[e], u2[e], u3[e]);
      } else {
#pragma unroll
        for (int e = 0; e < kElems; ++e) {
          const Split sp = split_double(x[e]);
          const unsigned long long a = quantise_abs(sp, ex, rn != 0);
          const unsigned long long t = sp.neg ? 0ull - a : a;
          const uint32_t lo = static_cast<uint32_t>(t);
          const int hi = static_cast<int>(t >> 32);
          b[e] = ((lo << 2) & 0x3FFFCu) | (4u * kDecBias);
          u1[e] = lo >> 16;
          u2[e] = static_cast<uint32_t>(hi) & 0xFFFFu;
          u3[e] = hi >> 16;
        }
      }
      planes_all(std::make_integer_sequence<int, R>{}, b, u1, u2, u3, table, dst);
    }
  }
}

static int num_sms() {
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return sms;
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
