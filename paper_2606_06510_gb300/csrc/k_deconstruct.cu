// Deconstruction (Algorithm 1 "lin:quant" and "lin:dec"; §2.5 digit planes)
// and the magnitude planes of the "+1" pass (§2.4).
//
// One thread handles 16 consecutive k-entries of one row of the operand
// (a row of A, or a column of B seen as a row of Bᵀ); the two threads of a
// lane pair cover 32 consecutive k-entries, so every plane row segment they
// write is one full 32-byte sector (16-byte vector stores).  A is column-
// major, so for A the 16 row-threads of a warp read 16 consecutive rows of
// one column per load (coalesced); B's rows are contiguous in k.
#include "oz2_common.cuh"

namespace oz2 {

constexpr int kElems = 16;               // k-entries per thread
constexpr int kRowsPerBlock = 128;       // 256 threads = 128 rows × 2 halves
constexpr int kDecThreads = 256;

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
};

// MODE 0: magnitude plane (1 plane); MODE 1: residue digit planes.
template <int MODE>
__global__ void __launch_bounds__(kDecThreads) planes_kernel(OperandView X, int64_t k, int64_t k_pad,
                                                             int clamp_c, int rn,
                                                             const __grid_constant__ Oz2Moduli mods,
                                                             const uint32_t* __restrict__ table_g) {
  extern __shared__ uint32_t table[];
  if (MODE == 1) {
    for (int t = threadIdx.x; t < mods.table_entries; t += blockDim.x) table[t] = table_g[t];
    __syncthreads();
  }
  const int64_t row_tiles = (X.rows + kRowsPerBlock - 1) / kRowsPerBlock;
  const int64_t k_tiles = k_pad / (2 * kElems);
  const int64_t ntiles = row_tiles * k_tiles;
  const int half = threadIdx.x & 1;
  const int rloc = threadIdx.x >> 1;
  const size_t plane_stride = static_cast<size_t>(X.rows) * k_pad;

  for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
    const int64_t kt = tile / row_tiles;  // consecutive blocks share a k-slice of many rows
    const int64_t rt = tile - kt * row_tiles;
    const int64_t row = rt * kRowsPerBlock + rloc;
    if (row >= X.rows) continue;
    const int64_t l0 = kt * (2 * kElems) + half * kElems;
    const uint8_t flag = X.flag[row];
    const int ex = X.exps[row];
    const bool zero_row = (flag & 2) != 0;
    uint8_t* dst = X.out + static_cast<size_t>(row) * k_pad + l0;

    if (MODE == 0) {
      uint32_t code[kElems];
#pragma unroll
      for (int e = 0; e < kElems; ++e) {
        int64_t l = l0 + e;
        code[e] = 0;
        if (!zero_row && l < k) {
          Split s = split_double(__ldg(X.base + row * X.row_stride + l * X.k_stride));
          if (s.M) code[e] = e4m3_pow2(max(-clamp_c, ceil_log2_abs(s) - ex));
        }
      }
      uint4 v;
      v.x = code[0] | (code[1] << 8) | (code[2] << 16) | (code[3] << 24);
      v.y = code[4] | (code[5] << 8) | (code[6] << 16) | (code[7] << 24);
      v.z = code[8] | (code[9] << 8) | (code[10] << 16) | (code[11] << 24);
      v.w = code[12] | (code[13] << 8) | (code[14] << 16) | (code[15] << 24);
      *reinterpret_cast<uint4*>(dst) = v;
    } else {
      // Quantise (Eq. scale) and split |Ã| into 16-bit limbs.
      uint32_t lo[kElems], hi[kElems];
      uint32_t negmask = 0;
#pragma unroll
      for (int e = 0; e < kElems; ++e) {
        int64_t l = l0 + e;
        unsigned long long a = 0;
        if (!zero_row && l < k) {
          Split s = split_double(__ldg(X.base + row * X.row_stride + l * X.k_stride));
          a = quantise_abs(s, ex, rn != 0);
          if (s.neg && a) negmask |= 1u << e;
        }
        lo[e] = static_cast<uint32_t>(a);
        hi[e] = static_cast<uint32_t>(a >> 32);
      }
#pragma unroll 1
      for (int i = 0; i < mods.r; ++i) {
        const uint32_t mi = static_cast<uint32_t>(mods.m[i]);
        const uint32_t mg = mods.magic[i];
        const int sh = mods.magic_sh[i];
        const uint32_t c1 = mods.limb[i][1], c2 = mods.limb[i][2], c3 = mods.limb[i][3];
        const uint32_t noff = static_cast<uint32_t>(mods.negoff[i]);
        const uint32_t* tab = table + mods.table_off[i];
        uint32_t w[kElems];
#pragma unroll
        for (int e = 0; e < kElems; ++e) {
          // |Ã| mod m from the limbs: y = u0 + u1·(2^16 mod m) + u2·(2^32 mod m) + u3·(2^48 mod m)
          uint32_t y = (lo[e] & 0xFFFFu) + (lo[e] >> 16) * c1 + (hi[e] & 0xFFFFu) * c2 +
                       (hi[e] >> 16) * c3;
          y = ((negmask >> e) & 1u) ? noff - y : y;  // residue of -|Ã|
          uint32_t r = mod_magic(y, mi, mg, sh);
          w[e] = tab[r];                              // packed E4M3 planes of centred(r)
        }
        const int np = mods.sq_base[i] ? 2 : 3;
        uint8_t* pdst = dst + static_cast<size_t>(mods.plane_off[i]) * plane_stride;
        for (int p = 0; p < np; ++p) {
          uint4 v;
          v.x = gather_byte(w[0], w[1], w[2], w[3], p);
          v.y = gather_byte(w[4], w[5], w[6], w[7], p);
          v.z = gather_byte(w[8], w[9], w[10], w[11], p);
          v.w = gather_byte(w[12], w[13], w[14], w[15], p);
          *reinterpret_cast<uint4*>(pdst + p * plane_stride) = v;
        }
      }
    }
  }
}

static int grid_for(int64_t rows, int64_t k_pad) {
  int64_t tiles = ((rows + kRowsPerBlock - 1) / kRowsPerBlock) * (k_pad / (2 * kElems));
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t cap = static_cast<int64_t>(sms) * 8;
  return static_cast<int>(tiles < cap ? (tiles > 0 ? tiles : 1) : cap);
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
  if (m > 0) {
    OperandView va{A, 1, lda, m, ra, row_flag, mag_a};
    count_launch();
    planes_kernel<0><<<grid_for(m, k_pad), kDecThreads, 0, st>>>(va, k, k_pad, c, 0, dummy, nullptr);
  }
  if (n > 0) {
    OperandView vb{B, ldb, 1, n, cb, col_flag, mag_b};
    count_launch();
    planes_kernel<0><<<grid_for(n, k_pad), kDecThreads, 0, st>>>(vb, k, k_pad, c, 0, dummy, nullptr);
  }
  return cudaGetLastError();
}

cudaError_t launch_deconstruct(int64_t m, int64_t n, int64_t k, const Oz2Moduli& mods,
                               const uint32_t* table_a, const uint32_t* table_b, const double* A, int64_t lda,
                               const double* B, int64_t ldb, const int32_t* d, const int32_t* e,
                               const uint8_t* row_flag, const uint8_t* col_flag, int quant,
                               uint8_t* planes_a, uint8_t* planes_b, cudaStream_t st) {
  const int64_t k_pad = (k + kKPad - 1) / kKPad * kKPad;
  size_t smem = sizeof(uint32_t) * mods.table_entries;
  cudaError_t err = cudaFuncSetAttribute(planes_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
  if (err != cudaSuccess) return err;
  const int rn = quant == OZ2_QUANT_RN;
  if (m > 0) {
    OperandView va{A, 1, lda, m, d, row_flag, planes_a};
    count_launch();
    planes_kernel<1><<<grid_for(m, k_pad), kDecThreads, smem, st>>>(va, k, k_pad, 0, rn, mods, table_a);
  }
  if (n > 0) {
    OperandView vb{B, ldb, 1, n, e, col_flag, planes_b};
    count_launch();
    planes_kernel<1><<<grid_for(n, k_pad), kDecThreads, smem, st>>>(vb, k, k_pad, 0, rn, mods, table_b);
  }
  return cudaGetLastError();
}

}  // namespace oz2
