// C ABI of liboz2 (declared in include/oz2.h): argument checks, the modulus
// constants and digit-plane table, workspace carving, and the stage order of
// Algorithm 1 (scan → "+1" pass and scales → deconstruct → residue GEMMs →
// Garner/unscale → native fallback).
#include <algorithm>
#include <cmath>
#include <atomic>
#include <cstdio>
#include <cstring>
#include <functional>
#include <mutex>
#include <vector>

#include "k_scan.cuh"

namespace oz2 {

// §2.5: the published set S (six squares, then the nonsquare tail), then the
// extension primes used for r = 13..16 (nonsquare, < 513).
static const int kModuliAll[kMaxModuli] = {1089, 1024, 961, 841, 625, 529, 511, 509,
                                           503,  499,  491, 487, 479, 467, 463, 461};
constexpr int kTableMax = 20480;  // 2·Σ of the ten nonsquare moduli = 9740 entries
constexpr int kHostBlocksMax = 8;   // column blocks of one oz2_dgemm_host call
constexpr int kHostAChunksMax = 4;  // column chunks A is copied in by oz2_dgemm_host

// Packed E4M3 digit planes of every residue (byte p = plane p) of the
// nonsquare moduli, 2m entries per modulus, entry i for the residue
// (i - kDecBias) mod m; table 0 for A (last plane pre-scaled by -16), table 1
// for B.
static __device__ uint32_t g_plane_table[2][kTableMax];
// Device status block (sticky status word, fallback counts, scale summary).
static __device__ Oz2Device g_status;

// ---------------------------------------------------------------------------
// Host-side arithmetic for the constants.
// ---------------------------------------------------------------------------
static int isqrt_exact(int m) {
  for (int s = 1; s * s <= m; ++s)
    if (s * s == m) return s;
  return 0;
}

// E4M3-exact integers: M·2^e with |M| ≤ 15 and magnitude ≤ 448 (§2.5).
static bool e4m3_exact(int v) {
  int a = v < 0 ? -v : v;
  if (a == 0) return true;
  if (a > 448) return false;
  while ((a & 1) == 0) a >>= 1;
  return a <= 15;
}

// E4M3 byte: sign | (e+7) << 3 | fraction, for an integer in 𝔼.
static uint8_t e4m3_code(int v) {
  if (v == 0) return 0;
  int a = v < 0 ? -v : v;
  int e = 31 - __builtin_clz(static_cast<unsigned>(a));
  int frac = ((a << 3) >> e) - 8;
  return static_cast<uint8_t>((v < 0 ? 0x80 : 0) | ((e + 7) << 3) | frac);
}

static int floor_mod(int a, int m) {
  int r = a % m;
  return r < 0 ? r + m : r;
}

// Digit planes of the centred residue d (§2.5).  With `merged` (the A
// operand) the last nonsquare plane is stored as -16·d1, the accumulator
// merge of §2.5: the products d0·e0 and (-16 d1)·e1 then share the weight
// (1 - 2^b) in one accumulator.
static uint32_t plane_word(int d, int m, bool merged) {
  int s = isqrt_exact(m);
  int p[3] = {0, 0, 0}, np;
  if (s) {  // balanced base s: d0 ∈ [-⌊s/2⌋, s-1-⌊s/2⌋]
    int h = s / 2;
    int d0 = floor_mod(d + h, s) - h;
    int d1 = (d - d0) / s;
    p[0] = d0;
    p[1] = d1;
    np = 2;
  } else {  // balanced base 16 with the carry correction
    int d0 = floor_mod(d + 8, 16) - 8;
    int d1 = (d - d0) / 16;
    if (!e4m3_exact(d0 + d1)) {
      int sg = d0 > 0 ? 1 : -1;
      d0 -= 16 * sg;
      d1 += sg;
    }
    p[0] = d0 + d1;
    p[1] = d0;
    p[2] = merged ? -16 * d1 : d1;
    np = 3;
  }
  uint32_t w = 0;
  for (int i = 0; i < np; ++i) {
    if (!e4m3_exact(p[i])) {
      std::fprintf(stderr, "oz2: digit %d of residue %d mod %d is not E4M3-exact\n", p[i], d, m);
      return 0xFFFFFFFFu;
    }
    w |= static_cast<uint32_t>(e4m3_code(p[i])) << (8 * i);
  }
  return w;
}

static int mod_inverse(long long a, int m) {
  long long t = 0, nt = 1, r = m, nr = floor_mod(static_cast<int>(a % m), m);
  while (nr) {
    long long q = r / nr, tmp;
    tmp = t - q * nt; t = nt; nt = tmp;
    tmp = r - q * nr; r = nr; nr = tmp;
  }
  return static_cast<int>(t < 0 ? t + m : t);
}

typedef unsigned long long u64;
static void mul3(u64 (&x)[3], u64 m) {
  unsigned __int128 c = 0;
  for (int i = 0; i < 3; ++i) {
    unsigned __int128 p = static_cast<unsigned __int128>(x[i]) * m + c;
    x[i] = static_cast<u64>(p);
    c = p >> 64;
  }
}
static int bitlen3(const u64 (&x)[3]) {
  for (int i = 2; i >= 0; --i)
    if (x[i]) return 64 * i + 64 - __builtin_clzll(x[i]);
  return 0;
}

// v = hi·2^32 + lo (mod 2^64) with lo the low word read as a signed integer.
static void split_signed_low(u64 v, int* lo, int* hi) {
  const int l = static_cast<int>(static_cast<uint32_t>(v));
  *lo = l;
  *hi = static_cast<int>(static_cast<uint32_t>((v - static_cast<u64>(static_cast<long long>(l))) >> 32));
}

static Oz2Moduli build_moduli(int r, int quant) {
  Oz2Moduli c;
  std::memset(&c, 0, sizeof(c));
  c.r = r;
  int plane = 0, toff = 0;
  for (int i = 0; i < r; ++i) {
    const int m = kModuliAll[i];
    c.m[i] = m;
    c.sq_base[i] = isqrt_exact(m);
    c.plane_off[i] = plane;
    plane += c.sq_base[i] ? 2 : 3;
    if (!c.sq_base[i]) toff += m;  // the digit-plane table holds nonsquare moduli only
    c.goff[i] = m * static_cast<int>(((1u << 27) + m - 1) / m);
    long long P = 1;  // product of the earlier moduli, mod m
    for (int t = 0; t < i; ++t) {
      c.pmod[i][t] = static_cast<int>(P);
      P = (P * kModuliAll[t]) % m;
    }
    c.inv[i] = i ? mod_inverse(P, m) : 1;
    c.invp[i] = static_cast<uint32_t>((static_cast<u64>(c.inv[i]) << 32) / static_cast<u64>(m));
  }
  c.nplanes = plane;
  c.table_entries = 2 * toff;
  // Direct-CRT constants.
  for (int k = 0; k < r; ++k) {
    const int mk = kModuliAll[k];
    uint32_t W[6] = {1, 0, 0, 0, 0, 0};  // Π_{j≠k} m_j, then × y_k
    long long pm = 1;                    // Π_{j≠k} m_j mod m_k
    for (int j = 0; j < r; ++j) {
      if (j == k) continue;
      u64 carry = 0;
      for (int t = 0; t < 6; ++t) {
        const u64 v = static_cast<u64>(W[t]) * static_cast<u64>(kModuliAll[j]) + carry;
        W[t] = static_cast<uint32_t>(v);
        carry = v >> 32;
      }
      pm = (pm * kModuliAll[j]) % mk;
    }
    const int y = mod_inverse(pm, mk);
    u64 carry = 0;
    for (int t = 0; t < 6; ++t) {
      const u64 v = static_cast<u64>(W[t]) * static_cast<u64>(y) + carry;
      W[t] = static_cast<uint32_t>(v);
      carry = v >> 32;
    }
    for (int t = 0; t < 5; ++t) c.crtw[k][t] = W[t];
    c.crtf[k] = static_cast<uint32_t>(((static_cast<u64>(y) << 32) + static_cast<u64>(mk / 2)) / static_cast<u64>(mk));
    c.coff[k] = mk * ((32768 + mk - 1) / mk);
    // Two-word constants: y/m < 1 - 1/m, so both roundings stay below 2^64 and 2^18.
    const unsigned __int128 fy = ((static_cast<unsigned __int128>(y) << 64) + static_cast<unsigned>(mk / 2)) / mk;
    split_signed_low(static_cast<u64>(fy), &c.crt_fl[k], &c.crt_fh[k]);
    split_signed_low(static_cast<u64>(W[0]) | (static_cast<u64>(W[1]) << 32), &c.crt_wl[k], &c.crt_wh[k]);
    c.crt_g[k] = static_cast<int>(((static_cast<u64>(y) << 18) + static_cast<u64>(mk / 2)) / static_cast<u64>(mk));
  }
  u64 M[3] = {1, 0, 0};
  for (int i = 0; i < r; ++i) mul3(M, static_cast<u64>(kModuliAll[i]));
  for (int i = 0; i < 3; ++i) c.M[i] = M[i];
  // 96-bit constants (the fused kernel, r = 11, 12, M < 2^112): F_k =
  // round(2^96·y_k/m_k) split into signed low words, and the error bound of
  // the estimate of |X|: |X| - ⌊|Y|·M/2^96⌋ (partial products below 2^64
  // dropped) is within (Σ_k ⌊m_k/2⌋)·M/2^97 + 5 <
  // (Σ ⌊m_k/2⌋)·(⌊M/2^64⌋ + 1)/2^33 + 5 for centred residues.
  {
    u64 sum_centred = 0;
    for (int k = 0; k < r; ++k) {
      const int mk = kModuliAll[k];
      long long pm = 1;
      for (int j = 0; j < r; ++j)
        if (j != k) pm = (pm * kModuliAll[j]) % mk;
      const int y = mod_inverse(pm, mk);
      const unsigned __int128 F = ((static_cast<unsigned __int128>(y) << 96) + static_cast<unsigned>(mk / 2)) / mk;
      int lo = 0, hi = 0;
      split_signed_low(static_cast<u64>(F), &lo, &hi);
      c.crt_y0[k] = lo;
      const unsigned __int128 F1 = (F - static_cast<unsigned __int128>(static_cast<__int128>(lo))) >> 32;
      split_signed_low(static_cast<u64>(F1), &lo, &hi);
      c.crt_y1[k] = lo;
      c.crt_y2[k] = static_cast<uint32_t>((F1 - static_cast<unsigned __int128>(static_cast<__int128>(lo))) >> 32);
      sum_centred += static_cast<u64>(mk / 2);
    }
    for (int i = 0; i < 4; ++i) c.crt_m32[i] = static_cast<uint32_t>(M[i >> 1] >> (32 * (i & 1)));
    const unsigned __int128 mh1 = static_cast<unsigned __int128>(M[1]) + 1;  // M < 2^128 here
    c.crt_err_centred = static_cast<u64>((sum_centred * mh1 + ((static_cast<unsigned __int128>(1) << 33) - 1)) >> 33) + 6;
  }
  split_signed_low(M[0], &c.crt_ml, &c.crt_mlh);
  // round(M/2^51), below 2^61 while M < 2^112 (r ≤ 12, the only use).
  split_signed_low(((M[0] >> 51) | (M[1] << 13)) + ((M[0] >> 50) & 1), &c.crt_m51l, &c.crt_m51h);
  // ⌈M/2⌉ = (M + 1) >> 1
  u64 Mp[3] = {M[0] + 1, M[1] + (M[0] + 1 == 0), M[2]};
  c.Mhalf[0] = (Mp[0] >> 1) | (Mp[1] << 63);
  c.Mhalf[1] = (Mp[1] >> 1) | (Mp[2] << 63);
  c.Mhalf[2] = Mp[2] >> 1;
  // TZ: largest T with 2^(T+1) < M, i.e. bitlen(M-1) - 2; RN two bits less.
  u64 Mm1[3] = {M[0] - 1, M[1] - (M[0] == 0), M[2]};
  int t_tz = bitlen3(Mm1) - 2;
  c.T = quant == OZ2_QUANT_RN ? t_tz - 2 : t_tz;
  return c;
}

// ---------------------------------------------------------------------------
// Per-device state: the plane table is uploaded once per device.
// ---------------------------------------------------------------------------
struct DeviceState {
  bool ready = false;
  uint32_t* table_a = nullptr;
  uint32_t* table_b = nullptr;
  Oz2Device* status = nullptr;
  // Stream-ordered pool for the workspaces and staging buffers the library
  // allocates itself; it keeps freed blocks for reuse (release threshold:
  // unlimited) until oz2_trim_memory.  Created by the first call that
  // allocates, so entry points that allocate nothing never create it.
  cudaMemPool_t pool = nullptr;
  bool pool_tried = false;
  // oz2_dgemm_host: a stream for the copies (A and B in, then the finished
  // column blocks of C back), one event for the staging buffer's
  // allocation, one per arrived part of the operands, one per block and one
  // for the last copy, created on first use; the mutex serialises
  // host-buffer calls on this device, which share them.
  std::mutex host_mu;
  cudaStream_t copy_stream = nullptr;
  cudaEvent_t staged = nullptr;
  cudaEvent_t arrived[1 + kHostAChunksMax] = {};
  cudaEvent_t block_done[kHostBlocksMax] = {};
  cudaEvent_t copies_done = nullptr;
};
static DeviceState g_devs[64];
static std::mutex g_mu;

// Per-stage timing: each timed call records 9 events into one set of a
// ring; sets are harvested (synchronised) when stats are read or when the
// ring wraps onto a set still pending.
constexpr int kTimingSets = 32;
struct TimingSet {
  cudaEvent_t ev[9];
  bool created = false;
  bool pending = false;
};
struct HostStats {
  int k_slab = 0;
  double stage_sum[8] = {0};
  int timed = 0;
  TimingSet sets[kTimingSets];
  int next = 0;
};
static HostStats g_host_stats[64];
static std::atomic<long long> g_launches{0};

static void harvest(HostStats& hs, TimingSet& t) {
  if (!t.pending) return;
  if (cudaEventSynchronize(t.ev[8]) == cudaSuccess) {
    for (int i = 0; i < 8; ++i) {
      float ms = 0.f;
      cudaEventElapsedTime(&ms, t.ev[i], t.ev[i + 1]);
      hs.stage_sum[i] += ms;
    }
    ++hs.timed;
  }
  t.pending = false;
}

static int device_state(DeviceState** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return OZ2_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_mu);
  DeviceState& s = g_devs[dev];
  if (!s.ready) {
    static uint32_t host_table[2][kTableMax];
    for (int t = 0; t < 2; ++t) {
      int off = 0;
      for (int i = 0; i < kMaxModuli; ++i) {
        const int m = kModuliAll[i];
        if (isqrt_exact(m)) continue;  // square moduli compute their digits
        for (int j = 0; j < 2 * m; ++j) {
          const int r = floor_mod(j - static_cast<int>(kDecBias % static_cast<uint32_t>(m)), m);
          const int d = r > m - 1 - m / 2 ? r - m : r;  // centred residue
          const uint32_t w = plane_word(d, m, t == 0);
          if (w == 0xFFFFFFFFu) return OZ2_ERR_CUDA;
          host_table[t][off + j] = w;
        }
        off += 2 * m;
      }
    }
    if (cudaMemcpyToSymbol(g_plane_table, host_table, sizeof(host_table)) != cudaSuccess) return OZ2_ERR_CUDA;
    Oz2Device zero;
    std::memset(&zero, 0, sizeof(zero));
    if (cudaMemcpyToSymbol(g_status, &zero, sizeof(zero)) != cudaSuccess) return OZ2_ERR_CUDA;
    uint32_t* tables = nullptr;
    if (cudaGetSymbolAddress(reinterpret_cast<void**>(&tables), g_plane_table) != cudaSuccess ||
        cudaGetSymbolAddress(reinterpret_cast<void**>(&s.status), g_status) != cudaSuccess)
      return OZ2_ERR_CUDA;
    s.table_a = tables;
    s.table_b = tables + kTableMax;
    s.ready = true;
  }
  *out = &s;
  return OZ2_OK;
}

// Stream-ordered allocation from the library's pool on the current device
// (the pool is created here, on the device's first allocation).
static cudaError_t pool_alloc(void** p, size_t bytes, cudaStream_t s) {
  DeviceState* ds = nullptr;
  if (device_state(&ds) != OZ2_OK) return cudaErrorInitializationError;
  {
    std::lock_guard<std::mutex> lk(g_mu);
    if (!ds->pool_tried) {
      ds->pool_tried = true;
      int dev = 0;
      cudaGetDevice(&dev);
      cudaMemPoolProps props;
      std::memset(&props, 0, sizeof(props));
      props.allocType = cudaMemAllocationTypePinned;
      props.location.type = cudaMemLocationTypeDevice;
      props.location.id = dev;
      if (cudaMemPoolCreate(&ds->pool, &props) == cudaSuccess) {
        cuuint64_t keep = ~cuuint64_t(0);
        cudaMemPoolSetAttribute(ds->pool, cudaMemPoolAttrReleaseThreshold, &keep);
      } else {
        cudaGetLastError();
        ds->pool = nullptr;  // the device's default pool serves instead
      }
    }
  }
  return ds->pool ? cudaMallocFromPoolAsync(p, bytes, ds->pool, s) : cudaMallocAsync(p, bytes, s);
}

// Column-major rows × cols matrix copy; one linear copy when both sides are
// contiguous (ld = rows), a pitched copy otherwise.
static cudaError_t copy_matrix(double* dst, int64_t dld, const double* src, int64_t sld, int64_t rows, int64_t cols,
                               cudaMemcpyKind kind, cudaStream_t s) {
  if (rows == 0 || cols == 0) return cudaSuccess;
  if ((dld == rows && sld == rows) || cols == 1)
    return cudaMemcpyAsync(dst, src, sizeof(double) * rows * cols, kind, s);
  return cudaMemcpy2DAsync(dst, sizeof(double) * dld, src, sizeof(double) * sld, sizeof(double) * rows, cols, kind,
                           s);
}

__global__ void reset_status_kernel(Oz2Device* dev) {
  dev->fallback_rows = 0;
  dev->fallback_cols = 0;
  dev->u_max_bits = 0;
  dev->s = 0;
}

// The start of a call: the status summary, and the workspace words that
// later stages accumulate with atomics (scan keys ra, cb; the "+1" row
// maxima; the two fallback counts) set to zero, in one launch.
__global__ void prepare_call_kernel(Oz2Device* dev, int* ra, int64_t m, int* cb, int64_t n, float* urow,
                                    int* counts) {
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    dev->fallback_rows = 0;
    dev->fallback_cols = 0;
    dev->u_max_bits = 0;
    dev->s = 0;
    counts[0] = 0;
    counts[1] = 0;
  }
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < m + n; i += (int64_t)gridDim.x * blockDim.x) {
    if (i < m) {
      ra[i] = 0;
      urow[i] = 0.f;
    } else {
      cb[i - m] = 0;
    }
  }
}

void count_launch(int n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

static size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

static void compute_layout(int64_t m, int64_t n, int64_t k, int r, oz2_ws_layout* L) {
  const int64_t k_pad = (k + kKPad - 1) / kKPad * kKPad;
  int planes = 0;
  for (int i = 0; i < r; ++i) planes += isqrt_exact(kModuliAll[i]) ? 2 : 3;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off = align256(off + bytes);
    return o;
  };
  L->ra = take(4 * m);
  L->cb = take(4 * n);
  L->row_flag = take(m);
  L->col_flag = take(n);
  L->d = take(4 * m);
  L->e = take(4 * n);
  L->urow = take(4 * m);
  L->misc = take(4 * (m + n + 2));
  L->mag_a = take(static_cast<size_t>(m) * k_pad);
  L->mag_b = take(static_cast<size_t>(n) * k_pad);
  // Digit planes in 128 × 128-byte blocks: rows padded to a multiple of 128.
  L->planes_a = take(static_cast<size_t>(planes) * ((m + 127) / 128 * 128) * k_pad);
  L->planes_b = take(static_cast<size_t>(planes) * ((n + 127) / 128 * 128) * k_pad);
  const int64_t res_ld = (m + 7) / 8 * 8;  // 16-byte columns
  L->residues = take(2 * static_cast<size_t>(r) * n * res_ld);
  L->total = off;
  L->k_pad = k_pad;
  L->num_planes = planes;
  L->res_ld = res_ld;
}

static int check_sizes(int64_t m, int64_t n, int64_t k, int64_t lda, int64_t ldb, int64_t ldc) {
  if (m < 0 || n < 0 || k < 0) return OZ2_ERR_INVALID_ARG;
  if (lda < std::max<int64_t>(1, m) || ldb < std::max<int64_t>(1, k) || ldc < std::max<int64_t>(1, m))
    return OZ2_ERR_INVALID_ARG;
  // Tile coordinates are 32-bit; U·2^2c ≤ k·2^2c ≤ 2^24 needs k ≤ 2^24.
  if (m >= (1LL << 31) || n >= (1LL << 31) || k > (1LL << 24)) return OZ2_ERR_UNSUPPORTED;
  return OZ2_OK;
}

static int to_status(cudaError_t e) { return e == cudaSuccess ? OZ2_OK : OZ2_ERR_CUDA; }

}  // namespace oz2

using namespace oz2;

extern "C" {

const char* oz2_status_string(int status) {
  switch (status) {
    case OZ2_OK: return "OZ2_OK";
    case OZ2_ERR_INVALID_ARG: return "OZ2_ERR_INVALID_ARG";
    case OZ2_ERR_UNSUPPORTED_R: return "OZ2_ERR_UNSUPPORTED_R";
    case OZ2_ERR_ALLOC: return "OZ2_ERR_ALLOC";
    case OZ2_ERR_CUDA: return "OZ2_ERR_CUDA";
    case OZ2_ERR_TIMEOUT: return "OZ2_ERR_TIMEOUT";
    case OZ2_ERR_UNSUPPORTED: return "OZ2_ERR_UNSUPPORTED";
    default: return "OZ2_ERR_UNKNOWN";
  }
}

int oz2_plane_layout(int num_moduli, int32_t* plane_offset) {
  if (num_moduli < 1 || num_moduli > kMaxModuli) return OZ2_ERR_UNSUPPORTED_R;
  int p = 0;
  for (int i = 0; i < num_moduli; ++i) {
    if (plane_offset) plane_offset[i] = p;
    p += isqrt_exact(kModuliAll[i]) ? 2 : 3;
  }
  return p;
}

size_t oz2_workspace_size(int64_t m, int64_t n, int64_t k, int num_moduli) {
  if (m < 0 || n < 0 || k < 0 || num_moduli < 1 || num_moduli > kMaxModuli) return 0;
  oz2_ws_layout L;
  compute_layout(m, n, k, num_moduli, &L);
  return L.total;
}

// Leading square moduli of the first r (the published set lists its squares
// first); the residue GEMM schedules the nonsquare ones before them.
static int leading_squares(int r) {
  int q = 0;
  while (q < r && isqrt_exact(kModuliAll[q])) ++q;
  return q;
}

int oz2_workspace_layout(int64_t m, int64_t n, int64_t k, int num_moduli, oz2_ws_layout* out) {
  if (!out || m < 0 || n < 0 || k < 0) return OZ2_ERR_INVALID_ARG;
  if (num_moduli < 1 || num_moduli > kMaxModuli) return OZ2_ERR_UNSUPPORTED_R;
  compute_layout(m, n, k, num_moduli, out);
  return OZ2_OK;
}

// Called after the stages of a column block [c0, c0 + cols) of C are
// enqueued on the call's stream.
typedef std::function<cudaError_t(int64_t c0, int64_t cols)> BlockDone;

// Column blocks of C: widths[0..count), each a multiple of 256 but the last.
struct ColumnBlocks {
  int count = 0;
  int64_t widths[kHostBlocksMax] = {};
};

// Operands that arrive on another stream while phase 1 runs (oz2_dgemm_host):
// B whole when b_ready has completed, then A by column chunks, columns
// [a_col0[c], a_col0[c + 1]) when a_ready[c] has.
struct Arrivals {
  cudaEvent_t b_ready = nullptr;
  int a_chunks = 0;
  int64_t a_col0[kHostAChunksMax + 1] = {};
  cudaEvent_t a_ready[kHostAChunksMax] = {};
};

// Algorithm 1 on the call's stream.  Phase 1 (scan, "+1" pass, scales,
// deconstruction) covers the whole problem; the residue GEMM, the
// reconstruction and the fallback then run per column block (all of C when
// `blocks` is null), each followed by `on_block`.  With `in`, the operands
// are still arriving: B's scan, flags and magnitude planes run as soon as B
// is in, and A's scan chunk by chunk as its columns come (the row keys are
// maxima, merged across chunks).  The results depend on neither.
static int run_stages(int64_t m, int64_t n, int64_t k, const double* A, int64_t lda, const double* B, int64_t ldb,
                      double* C, int64_t ldc, int num_moduli, int quant, int scale, unsigned flags, void* workspace,
                      size_t ws_bytes, void* stream, const ColumnBlocks* blocks, const BlockDone* on_block,
                      const Arrivals* in = nullptr) {
  int st = check_sizes(m, n, k, lda, ldb, ldc);
  if (st) return st;
  if (num_moduli < 1 || num_moduli > kMaxModuli) return OZ2_ERR_UNSUPPORTED_R;
  if ((quant != OZ2_QUANT_TZ && quant != OZ2_QUANT_RN) || (scale != OZ2_SCALE_R2 && scale != OZ2_SCALE_R1))
    return OZ2_ERR_INVALID_ARG;
  if (m == 0 || n == 0) return OZ2_OK;
  if (!C || (k > 0 && (!A || !B))) return OZ2_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (k == 0) return to_status(cudaMemset2DAsync(C, ldc * sizeof(double), 0, m * sizeof(double), n, s));

  oz2_ws_layout L;
  compute_layout(m, n, k, num_moduli, &L);
  if (!workspace || ws_bytes < L.total || (reinterpret_cast<uintptr_t>(workspace) & 255)) return OZ2_ERR_ALLOC;
  DeviceState* ds = nullptr;
  if ((st = device_state(&ds)) != OZ2_OK) return st;
  const Oz2Moduli mods = build_moduli(num_moduli, quant);

  uint8_t* ws = static_cast<uint8_t*>(workspace);
  int32_t* ra = reinterpret_cast<int32_t*>(ws + L.ra);
  int32_t* cb = reinterpret_cast<int32_t*>(ws + L.cb);
  uint8_t* rf = ws + L.row_flag;
  uint8_t* cf = ws + L.col_flag;
  int32_t* d = reinterpret_cast<int32_t*>(ws + L.d);
  int32_t* e = reinterpret_cast<int32_t*>(ws + L.e);
  float* urow = reinterpret_cast<float*>(ws + L.urow);
  int* misc = reinterpret_cast<int*>(ws + L.misc);
  uint8_t* mag_a = ws + L.mag_a;
  uint8_t* mag_b = ws + L.mag_b;
  uint8_t* pa = ws + L.planes_a;
  uint8_t* pb = ws + L.planes_b;
  int16_t* res = reinterpret_cast<int16_t*>(ws + L.residues);

  const bool timing = (flags & OZ2_FLAG_TIMING) != 0;
  const bool simt = (flags & OZ2_FLAG_DEBUG_SIMT_GEMM) != 0;
  // On request, for short k: the residue GEMM and the reconstruction fused,
  // the residues kept on chip; the residue region then holds the fused
  // kernel's list of outputs left to the exact reconstruction.
  const bool fused = !simt && (flags & OZ2_FLAG_FUSED) != 0 && fused_crt_applies(L.k_pad, num_moduli);
  // A skinny C: A's digit planes formed on chip inside the residue GEMM
  // (never stored), only B deconstructed ahead.
  const bool onfly = !simt && !fused && (flags & OZ2_FLAG_ON_THE_FLY) != 0 && modef_applies(m, n, L.k_pad);
  int dev = 0;
  cudaGetDevice(&dev);
  HostStats& hs = g_host_stats[dev];
  TimingSet* ts = nullptr;
  if (timing) {
    std::lock_guard<std::mutex> lk(g_mu);
    ts = &hs.sets[hs.next];
    hs.next = (hs.next + 1) % kTimingSets;
    harvest(hs, *ts);
    if (!ts->created) {
      for (int i = 0; i < 9; ++i) cudaEventCreate(&ts->ev[i]);
      ts->created = true;
    }
  }
  auto mark = [&](int i) {
    if (ts) cudaEventRecord(ts->ev[i], s);
  };

  cudaError_t err = cudaSuccess;
  count_launch();
  {
    const int64_t blocks = std::min<int64_t>((m + n + 255) / 256, 1024);
    prepare_call_kernel<<<static_cast<unsigned>(std::max<int64_t>(blocks, 1)), 256, 0, s>>>(ds->status, ra, m, cb,
                                                                                              n, urow, misc);
  }
  mark(0);
  const ScanOut so{ra, cb, rf, cf};
  if (in) {
    if (err == cudaSuccess) err = cudaStreamWaitEvent(s, in->b_ready, 0);
    if (err == cudaSuccess) err = launch_scan_keys(0, n, k, nullptr, lda, B, ldb, so, s);
    if (err == cudaSuccess) err = launch_scan_flags(m, n, 2, flags, so, ds->status, s);
    if (err == cudaSuccess && scale == OZ2_SCALE_R2)
      err = launch_magnitude_planes(0, n, k, A, lda, B, ldb, ra, cb, rf, cf, mag_a, mag_b, s);
    for (int c = 0; c < in->a_chunks && err == cudaSuccess; ++c) {
      err = cudaStreamWaitEvent(s, in->a_ready[c], 0);
      const int64_t k0 = in->a_col0[c];
      if (err == cudaSuccess)
        err = launch_scan_keys(m, 0, in->a_col0[c + 1] - k0, A + k0 * lda, lda, nullptr, ldb, so, s);
    }
    if (err == cudaSuccess) err = launch_scan_flags(m, n, 1, flags, so, ds->status, s);
  } else if (err == cudaSuccess) {
    err = launch_scan(m, n, k, A, lda, B, ldb, flags, so, ds->status, s, false);
  }
  mark(1);
  if (scale == OZ2_SCALE_R2) {
    if (err == cudaSuccess)
      err = launch_magnitude_planes(m, in ? 0 : n, k, A, lda, B, ldb, ra, cb, rf, cf, mag_a, mag_b, s);
    mark(2);
    // The digit-plane and residue regions are not yet in use: the scratch
    // for the magnitude GEMM's partial sums when it splits k.
    if (err == cudaSuccess)
      err = launch_plane_gemm(m, n, L.k_pad, mods, mag_a, mag_b, simt ? 3 : 1, nullptr, 0, urow, ds->status, s,
                              reinterpret_cast<int16_t*>(pa), L.total - L.planes_a);
    mark(3);
  } else {
    mark(2);
    mark(3);
  }
  if (err == cudaSuccess) err = launch_choose_scales(m, n, k, mods, scale, urow, ra, cb, rf, cf, d, e, ds->status, s);
  mark(4);
  if (err == cudaSuccess)
    err = launch_deconstruct(onfly ? 0 : m, n, k, mods, ds->table_a, ds->table_b, A, lda, B, ldb, d, e, rf, cf, quant,
                             pa, pb, s);
  mark(5);
  // Phase 2 by column blocks (stage timing needs a single block).
  const bool blocked = blocks && blocks->count > 1 && !ts;
  const int nblk = blocked ? blocks->count : 1;
  int64_t c0 = 0;
  for (int bi = 0; bi < nblk && err == cudaSuccess; ++bi) {
    const int64_t cols = blocked ? blocks->widths[bi] : n;
    const uint8_t* pb0 = pb + static_cast<size_t>(c0 / kPlaneRows) * (L.k_pad / kPlaneLine) * L.num_planes *
                                  static_cast<size_t>(kPlaneBlock);
    if (fused) {
      err = launch_fused_crt(m, cols, L.k_pad, mods, pa, pb0, d, e + c0, rf, cf + c0, C + c0 * ldc, ldc, res,
                             L.total - L.residues, ds->status, s);
      mark(6);
      mark(7);
    } else {
      if (onfly) {
        err = launch_modef(m, cols, k, mods, ds->table_a, A, lda, d, rf, quant, pb0, res, L.res_ld, ds->status, s);
      } else {
        // The magnitude planes are dead once the scales are chosen: their
        // region is the scratch for the partial residues of a split-K GEMM.
        err = launch_plane_gemm(m, cols, L.k_pad, mods, pa, pb0, simt ? 2 : 0, res, L.res_ld, nullptr, ds->status, s,
                                reinterpret_cast<int16_t*>(mag_a), L.planes_a - L.mag_a);
      }
      mark(6);
      if (err == cudaSuccess)
        err = launch_reconstruct(m, cols, mods, res, L.res_ld, d, e + c0, C + c0 * ldc, ldc, s);
      mark(7);
    }
    if (err == cudaSuccess)
      err = launch_fallback_lists(m, cols, k, A, lda, B + c0 * ldb, ldb, rf, cf + c0, misc, C + c0 * ldc, ldc, s,
                                  c0 > 0);
    mark(8);
    if (err == cudaSuccess && on_block) err = (*on_block)(c0, cols);
    c0 += cols;
  }

  hs.k_slab = static_cast<int>(std::min<int64_t>(kKSlabMerged, L.k_pad));
  if (ts) ts->pending = true;
  return to_status(err);
}

int oz2_dgemm_ex(int64_t m, int64_t n, int64_t k, const double* A, int64_t lda, const double* B, int64_t ldb,
                 double* C, int64_t ldc, int num_moduli, int quant, int scale, unsigned flags, void* workspace,
                 size_t ws_bytes, void* stream) {
  return run_stages(m, n, k, A, lda, B, ldb, C, ldc, num_moduli, quant, scale, flags, workspace, ws_bytes, stream,
                    nullptr, nullptr);
}

// Column blocks for oz2_dgemm_host, chosen on a model of the call's second
// phase.  Block i's residue GEMM takes ⌈u_i/P⌉ waves of one unit's time
// (u_i = ⌈m/256⌉·r units per tile column of the block, P CTA pairs), its
// reconstruction moves m·(2r + 8) bytes of HBM per column, and its copy back
// moves 8m bytes per column over the host link, on one stream, once the
// block is done and the copy before it has finished.  Among the partitions
// into at most kHostBlocksMax blocks of whole tile columns (or of groups of
// them, when C has more than 64), the one whose last copy ends first is
// taken, by dynamic programming over the Pareto front of (end of compute,
// end of copies) after each prefix of the columns.  A small first block
// starts the copies early when the link is the bottleneck (short k); a
// small last block leaves little copy exposed when the GPU is (long k).
// The rates are this kernel's, measured on one GB300 and its host link.
namespace {
constexpr double kModelPairFlops = 46e12;     // residue GEMM, FP8 flop/s per CTA pair
constexpr double kModelUnitExtra = 2e-6;      // per unit: the accumulator drain
constexpr double kModelCrtBytes = 4.0e12;     // reconstruction, bytes/s
constexpr double kModelLink = 190e9;          // device to pinned host, bytes/s
constexpr double kModelBlockExtra = 8e-6;     // per block: its launches
constexpr double kModelCopyExtra = 5e-6;      // per copy
constexpr int kModelGroupsMax = 64;

struct BlockModel {
  int64_t m, n, tiles, per_tile, pairs, group;
  double t_unit, crt_per_col, d2h_per_col;
  int64_t cols(int64_t g0, int64_t g1) const {
    return std::min(n, g1 * group * 256) - std::min(n, g0 * group * 256);
  }
  double compute(int64_t g0, int64_t g1) const {
    const int64_t t = std::min(tiles, g1 * group) - g0 * group;
    const int64_t waves = (per_tile * t + pairs - 1) / pairs;
    return static_cast<double>(waves) * t_unit + static_cast<double>(cols(g0, g1)) * crt_per_col +
           kModelBlockExtra;
  }
  double copy(int64_t g0, int64_t g1) const { return static_cast<double>(cols(g0, g1)) * d2h_per_col + kModelCopyExtra; }
};

struct ModelState {
  double ce, cp;    // end of the blocks' compute, end of their copies
  int64_t g;        // groups covered
  int parent;       // index in the previous layer's front for g's predecessor
  int64_t from;     // first group of the last block
};
}  // namespace

static ColumnBlocks plan_column_blocks(int64_t m, int64_t n, int r, int64_t k, int64_t pairs) {
  ColumnBlocks b;
  const int64_t tiles = (n + 255) / 256;
  if (tiles < 2 || m == 0 || k == 0) {
    b.count = 1;
    b.widths[0] = n;
    return b;
  }
  BlockModel M;
  M.m = m;
  M.n = n;
  M.tiles = tiles;
  M.per_tile = (m + 255) / 256 * r;
  M.pairs = std::max<int64_t>(1, pairs);
  M.group = (tiles + kModelGroupsMax - 1) / kModelGroupsMax;
  const int64_t k_pad = (k + kKPad - 1) / kKPad * kKPad;
  M.t_unit = 3.0 * 2.0 * 256.0 * 256.0 * static_cast<double>(k_pad) / kModelPairFlops + kModelUnitExtra;
  M.crt_per_col = static_cast<double>(m) * (2.0 * r + 8.0) / kModelCrtBytes;
  M.d2h_per_col = static_cast<double>(m) * 8.0 / kModelLink;
  const int64_t G = (tiles + M.group - 1) / M.group;
  // fronts[j][g]: partitions of the first g groups into j blocks.
  std::vector<std::vector<std::vector<ModelState>>> fronts(
      kHostBlocksMax + 1, std::vector<std::vector<ModelState>>(G + 1));
  fronts[0][0].push_back(ModelState{0.0, 0.0, 0, -1, 0});
  double best = 1e300;
  int best_j = 0, best_i = 0;
  for (int j = 0; j <= kHostBlocksMax; ++j) {
    for (int64_t g = 0; g <= G; ++g) {
      std::vector<ModelState>& f = fronts[j][g];
      if (f.empty()) continue;
      // Keep the Pareto front: by compute end, then strictly falling copy end.
      std::sort(f.begin(), f.end(), [](const ModelState& x, const ModelState& y) {
        return x.ce < y.ce || (x.ce == y.ce && x.cp < y.cp);
      });
      std::vector<ModelState> kept;
      for (const ModelState& x : f)
        if (kept.empty() || x.cp < kept.back().cp) kept.push_back(x);
      f.swap(kept);
      if (g == G) {
        for (int i = 0; i < static_cast<int>(f.size()); ++i)
          if (f[i].cp < best - 1e-12) {
            best = f[i].cp;
            best_j = j;
            best_i = i;
          }
        continue;
      }
      if (j == kHostBlocksMax) continue;
      for (int i = 0; i < static_cast<int>(f.size()); ++i)
        for (int64_t g1 = g + 1; g1 <= G; ++g1) {
          const double ce = f[i].ce + M.compute(g, g1);
          const double cp = std::max(ce, f[i].cp) + M.copy(g, g1);
          fronts[j + 1][g1].push_back(ModelState{ce, cp, g1, i, g});
        }
    }
  }
  // Walk back from the best complete partition.
  int64_t widths[kHostBlocksMax];
  int j = best_j, i = best_i;
  int64_t g = G;
  while (j > 0) {
    const ModelState& x = fronts[j][g][i];
    widths[j - 1] = M.cols(x.from, g);
    i = x.parent;
    g = x.from;
    --j;
  }
  b.count = best_j;
  for (int q = 0; q < best_j; ++q) b.widths[q] = widths[q];
  return b;
}

// The plan of the last shape asked for is kept: a loop of calls on one shape
// plans once (a plan over many tile columns takes a few milliseconds).
static ColumnBlocks host_column_blocks(int64_t m, int64_t n, int r, int64_t k, int64_t pairs) {
  static std::mutex mu;
  static int64_t key[5] = {-1, -1, -1, -1, -1};
  static ColumnBlocks cached;
  const int64_t want[5] = {m, n, static_cast<int64_t>(r), k, pairs};
  std::lock_guard<std::mutex> lk(mu);
  if (!std::equal(want, want + 5, key)) {
    cached = plan_column_blocks(m, n, r, k, pairs);
    std::copy(want, want + 5, key);
  }
  return cached;
}

int oz2_plan(int64_t m, int64_t n, int64_t k, int num_moduli, int cta_pairs, oz2_plan_info* out) {
  if (!out || m < 0 || n < 0 || k < 0 || cta_pairs < 1) return OZ2_ERR_INVALID_ARG;
  if (num_moduli < 1 || num_moduli > kMaxModuli) return OZ2_ERR_UNSUPPORTED_R;
  *out = oz2_plan_info{};
  oz2_ws_layout L;
  compute_layout(m, n, k, num_moduli, &L);
  // The split-K scratch is the magnitude-plane region (dead by then).
  auto kparts = [&](int64_t cols) -> int64_t {
    if (m == 0 || cols == 0 || k == 0) return 1;
    return residue_gemm_kparts(m, cols, L.k_pad, num_moduli, leading_squares(num_moduli), L.res_ld,
                               L.planes_a - L.mag_a, cta_pairs);
  };
  out->kparts = kparts(n);
  out->mag_kparts = m > 0 && n > 0 && k > 0 ? magnitude_gemm_kparts(m, n, L.k_pad, L.total - L.planes_a, cta_pairs) : 1;
  const ColumnBlocks b = host_column_blocks(m, n, num_moduli, k, cta_pairs);
  out->host_blocks = b.count;
  for (int i = 0; i < b.count; ++i) {
    out->host_widths[i] = b.widths[i];
    out->host_kparts[i] = kparts(b.widths[i]);
  }
  return OZ2_OK;
}

int oz2_dgemm(int64_t m, int64_t n, int64_t k, const double* A, int64_t lda, const double* B, int64_t ldb,
              double* C, int64_t ldc, int num_moduli, void* stream) {
  int st = check_sizes(m, n, k, lda, ldb, ldc);
  if (st) return st;
  if (num_moduli < 1 || num_moduli > kMaxModuli) return OZ2_ERR_UNSUPPORTED_R;
  if (m == 0 || n == 0 || k == 0)
    return oz2_dgemm_ex(m, n, k, A, lda, B, ldb, C, ldc, num_moduli, OZ2_QUANT_TZ, OZ2_SCALE_R2, 0, nullptr, 0,
                        stream);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  size_t bytes = oz2_workspace_size(m, n, k, num_moduli);
  void* ws = nullptr;
  if (pool_alloc(&ws, bytes, s) != cudaSuccess) {
    cudaGetLastError();
    return OZ2_ERR_ALLOC;
  }
  st = oz2_dgemm_ex(m, n, k, A, lda, B, ldb, C, ldc, num_moduli, OZ2_QUANT_TZ, OZ2_SCALE_R2, 0, ws, bytes, stream);
  cudaError_t e2 = cudaFreeAsync(ws, s);
  if (st == OZ2_OK && e2 != cudaSuccess) st = OZ2_ERR_CUDA;
  return st;
}

int oz2_dgemm_host(int64_t m, int64_t n, int64_t k, const double* hA, int64_t lda, const double* hB, int64_t ldb,
                   double* hC, int64_t ldc, int num_moduli, void* stream) {
  int st = check_sizes(m, n, k, lda, ldb, ldc);
  if (st) return st;
  if (num_moduli < 1 || num_moduli > kMaxModuli) return OZ2_ERR_UNSUPPORTED_R;
  if (m == 0 || n == 0) return OZ2_OK;
  if (!hC || (k > 0 && (!hA || !hB))) return OZ2_ERR_INVALID_ARG;
  DeviceState* ds = nullptr;
  if ((st = device_state(&ds)) != OZ2_OK) return st;
  std::lock_guard<std::mutex> host_lock(ds->host_mu);
  if (!ds->copy_stream) {
    if (cudaStreamCreateWithFlags(&ds->copy_stream, cudaStreamNonBlocking) != cudaSuccess) return OZ2_ERR_CUDA;
    bool ok = cudaEventCreateWithFlags(&ds->staged, cudaEventDisableTiming) == cudaSuccess &&
              cudaEventCreateWithFlags(&ds->copies_done, cudaEventDisableTiming) == cudaSuccess;
    for (int i = 0; ok && i < 1 + kHostAChunksMax; ++i)
      ok = cudaEventCreateWithFlags(&ds->arrived[i], cudaEventDisableTiming) == cudaSuccess;
    for (int i = 0; ok && i < kHostBlocksMax; ++i)
      ok = cudaEventCreateWithFlags(&ds->block_done[i], cudaEventDisableTiming) == cudaSuccess;
    if (!ok) return OZ2_ERR_CUDA;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaStream_t cs = ds->copy_stream;
  const size_t bA = align256(sizeof(double) * m * k), bB = align256(sizeof(double) * k * n),
               bC = align256(sizeof(double) * m * n);
  const size_t ws = k > 0 ? oz2_workspace_size(m, n, k, num_moduli) : 0;
  uint8_t* buf = nullptr;
  if (pool_alloc(reinterpret_cast<void**>(&buf), bA + bB + bC + ws, s) != cudaSuccess) {
    cudaGetLastError();
    return OZ2_ERR_ALLOC;
  }
  double* dA = reinterpret_cast<double*>(buf);
  double* dB = reinterpret_cast<double*>(buf + bA);
  double* dC = reinterpret_cast<double*>(buf + bA + bB);
  // Every copy runs on the copy stream, after the staging buffer exists: B
  // first, then A by column chunks (of at least 32 MB, multiples of 64
  // columns), each marked by an event that the call's stream waits on
  // before the scan of that part (phase 1 overlaps the copies).
  cudaError_t err = cudaEventRecord(ds->staged, s);
  if (err == cudaSuccess) err = cudaStreamWaitEvent(cs, ds->staged, 0);
  Arrivals in;
  if (k > 0 && err == cudaSuccess) {
    err = copy_matrix(dB, k, hB, ldb, k, n, cudaMemcpyHostToDevice, cs);
    if (err == cudaSuccess) err = cudaEventRecord(ds->arrived[0], cs);
    in.b_ready = ds->arrived[0];
    const int64_t want = std::min<int64_t>(kHostAChunksMax, std::max<int64_t>(1, static_cast<int64_t>(bA >> 25)));
    const int64_t step = std::max<int64_t>(64, (k + want - 1) / want + 63) / 64 * 64;
    for (int64_t k0 = 0; k0 < k && err == cudaSuccess; k0 += step) {
      const int64_t kc = std::min(step, k - k0);
      err = copy_matrix(dA + k0 * m, m, hA + k0 * lda, lda, m, kc, cudaMemcpyHostToDevice, cs);
      if (err == cudaSuccess) err = cudaEventRecord(ds->arrived[1 + in.a_chunks], cs);
      in.a_ready[in.a_chunks] = ds->arrived[1 + in.a_chunks];
      in.a_col0[in.a_chunks++] = k0;
      in.a_col0[in.a_chunks] = k0 + kc;
    }
  }
  // C goes back by column blocks on the copy stream, each as soon as its
  // reconstruction and fallback are done, so that the copies overlap the
  // residue GEMM of the blocks after it.
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const ColumnBlocks blocks = host_column_blocks(m, n, num_moduli, k, std::max(1, sms / 2));
  int blk = 0;
  const BlockDone copy_back = [&](int64_t c0, int64_t cols) -> cudaError_t {
    cudaError_t e = cudaEventRecord(ds->block_done[blk], s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(cs, ds->block_done[blk], 0);
    if (e == cudaSuccess) e = copy_matrix(hC + c0 * ldc, ldc, dC + c0 * m, m, m, cols, cudaMemcpyDeviceToHost, cs);
    ++blk;
    return e;
  };
  if (err == cudaSuccess) {
    if (k > 0) {
      st = run_stages(m, n, k, dA, m, dB, k, dC, m, num_moduli, OZ2_QUANT_TZ, OZ2_SCALE_R2, 0,
                      buf + bA + bB + bC, ws, stream, &blocks, &copy_back, &in);
    } else {  // C = 0
      err = cudaMemsetAsync(dC, 0, sizeof(double) * m * n, s);
      if (err == cudaSuccess) err = copy_back(0, n);
    }
  }
  // The buffers are released once the copies have read them.
  if (cudaEventRecord(ds->copies_done, cs) == cudaSuccess) cudaStreamWaitEvent(s, ds->copies_done, 0);
  cudaFreeAsync(buf, s);
  if (cudaStreamSynchronize(s) != cudaSuccess && err == cudaSuccess) err = cudaErrorUnknown;
  if (st != OZ2_OK) return st;
  return to_status(err);
}

int oz2_trim_memory(void) {
  DeviceState* ds = nullptr;
  const int st = device_state(&ds);
  if (st) return st;
  if (cudaDeviceSynchronize() != cudaSuccess) return OZ2_ERR_CUDA;
  if (ds->pool && cudaMemPoolTrimTo(ds->pool, 0) != cudaSuccess) return OZ2_ERR_CUDA;
  return OZ2_OK;
}

int oz2_get_stats(oz2_stats* out) {
  if (!out) return OZ2_ERR_INVALID_ARG;
  DeviceState* ds = nullptr;
  int st = device_state(&ds);
  if (st) return st;
  if (cudaDeviceSynchronize() != cudaSuccess) return OZ2_ERR_CUDA;
  Oz2Device h;
  if (cudaMemcpy(&h, ds->status, sizeof(h), cudaMemcpyDeviceToHost) != cudaSuccess) return OZ2_ERR_CUDA;
  int dev = 0;
  cudaGetDevice(&dev);
  std::memset(out, 0, sizeof(*out));
  out->status = h.status ? OZ2_ERR_TIMEOUT : OZ2_OK;
  out->fallback_rows = h.fallback_rows;
  out->fallback_cols = h.fallback_cols;
  float u;
  std::memcpy(&u, &h.u_max_bits, sizeof(u));
  int ue = 0;
  if (u > 0.f) {
    unsigned b;
    std::memcpy(&b, &u, sizeof(b));
    ue = static_cast<int>((b >> 23) & 0xFF) - 127 + ((b & 0x7FFFFFu) ? 1 : 0);
  }
  out->u_max = ue;
  out->s = h.s;
  HostStats& hs = g_host_stats[dev];
  {
    std::lock_guard<std::mutex> lk(g_mu);
    for (int i = 0; i < kTimingSets; ++i) harvest(hs, hs.sets[i]);
    out->k_slab = hs.k_slab;
    out->timed_calls = hs.timed;
    for (int i = 0; i < 8; ++i) out->stage_ms[i] = hs.timed ? static_cast<float>(hs.stage_sum[i] / hs.timed) : 0.f;
    for (int i = 0; i < 8; ++i) hs.stage_sum[i] = 0;
    hs.timed = 0;
  }
  out->kernel_launches = g_launches.exchange(0);
  return OZ2_OK;
}

namespace oz2 {
// One warp waits on an mbarrier that nothing arrives at, bounded by `limit`
// SM cycles, and on expiry records the timeout as every library kernel does.
__global__ void timeout_probe_kernel(Oz2Device* dev, long long limit) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    const uint32_t b = smem_u32(&bar);
    mbar_init(b, 1);
    fence_barrier_init();
    if (!mbar_wait_bounded(b, 0, limit)) {
      dev->status = kStatusTimeout;
      dev->timeout_site = 9;
    }
  }
}
}  // namespace oz2

int oz2_selftest_timeout(long long limit_cycles, void* stream) {
  if (limit_cycles < 1000 || limit_cycles > 4000000000LL) return OZ2_ERR_INVALID_ARG;
  DeviceState* ds = nullptr;
  const int st = device_state(&ds);
  if (st) return st;
  count_launch();
  timeout_probe_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(ds->status, limit_cycles);
  return to_status(cudaGetLastError());
}

int oz2_probe_mma_rate(int64_t iters, int* cta_pairs, void* stream) {
  if (iters < 1 || iters > (int64_t{1} << 40)) return OZ2_ERR_INVALID_ARG;
  DeviceState* ds = nullptr;
  const int st = device_state(&ds);
  if (st) return st;
  return to_status(launch_mma_rate(iters, ds->status, cta_pairs, static_cast<cudaStream_t>(stream)));
}

int oz2_check_device_status(void) {
  DeviceState* ds = nullptr;
  int st = device_state(&ds);
  if (st) return st;
  if (cudaDeviceSynchronize() != cudaSuccess) return OZ2_ERR_CUDA;
  int v = 0;
  if (cudaMemcpy(&v, ds->status, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return OZ2_ERR_CUDA;
  if (v) {
    int zero = 0;
    cudaMemcpy(ds->status, &zero, sizeof(int), cudaMemcpyHostToDevice);
    return OZ2_ERR_TIMEOUT;
  }
  return OZ2_OK;
}

// ----------------------------- stage entry points ---------------------------
int oz2_scan(int64_t m, int64_t n, int64_t k, const double* A, int64_t lda, const double* B, int64_t ldb,
             unsigned flags, int32_t* ra, int32_t* cb, uint8_t* row_flag, uint8_t* col_flag, void* stream) {
  int st = check_sizes(m, n, k, lda, ldb, std::max<int64_t>(1, m));
  if (st) return st;
  if ((m && (!ra || !row_flag)) || (n && (!cb || !col_flag)) || (k && m && !A) || (k && n && !B))
    return OZ2_ERR_INVALID_ARG;
  DeviceState* ds = nullptr;
  if ((st = device_state(&ds)) != OZ2_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  count_launch();
  reset_status_kernel<<<1, 1, 0, s>>>(ds->status);
  return to_status(
      launch_scan(m, n, k, A, lda, B, ldb, flags, ScanOut{ra, cb, row_flag, col_flag}, ds->status, s, true));
}

int oz2_scale(int64_t m, int64_t n, int64_t k, int num_moduli, const double* A, int64_t lda, const double* B,
              int64_t ldb, const int32_t* ra, const int32_t* cb, const uint8_t* row_flag, const uint8_t* col_flag,
              int quant, int scale, uint8_t* mag_a, uint8_t* mag_b, float* urow, int32_t* d, int32_t* e,
              void* stream) {
  int st = check_sizes(m, n, k, lda, ldb, std::max<int64_t>(1, m));
  if (st) return st;
  if (num_moduli < 1 || num_moduli > kMaxModuli) return OZ2_ERR_UNSUPPORTED_R;
  if (m == 0 || n == 0 || k == 0) return OZ2_ERR_INVALID_ARG;
  if (!A || !B || !ra || !cb || !row_flag || !col_flag || !mag_a || !mag_b || !urow || !d || !e)
    return OZ2_ERR_INVALID_ARG;
  DeviceState* ds = nullptr;
  if ((st = device_state(&ds)) != OZ2_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const Oz2Moduli mods = build_moduli(num_moduli, quant);
  const int64_t k_pad = (k + kKPad - 1) / kKPad * kKPad;
  count_launch();
  reset_status_kernel<<<1, 1, 0, s>>>(ds->status);
  cudaError_t err = cudaMemsetAsync(urow, 0, sizeof(float) * m, s);
  if (scale == OZ2_SCALE_R2) {
    if (err == cudaSuccess)
      err = launch_magnitude_planes(m, n, k, A, lda, B, ldb, ra, cb, row_flag, col_flag, mag_a, mag_b, s);
    if (err == cudaSuccess)
      err = launch_plane_gemm(m, n, k_pad, mods, mag_a, mag_b, 1, nullptr, 0, urow, ds->status, s);
  }
  if (err == cudaSuccess)
    err = launch_choose_scales(m, n, k, mods, scale, urow, ra, cb, row_flag, col_flag, d, e, ds->status, s);
  return to_status(err);
}

int oz2_deconstruct(int64_t m, int64_t n, int64_t k, int num_moduli, const double* A, int64_t lda, const double* B,
                    int64_t ldb, const int32_t* d, const int32_t* e, const uint8_t* row_flag, const uint8_t* col_flag,
                    int quant, uint8_t* planes_a, uint8_t* planes_b, void* stream) {
  int st = check_sizes(m, n, k, lda, ldb, std::max<int64_t>(1, m));
  if (st) return st;
  if (num_moduli < 1 || num_moduli > kMaxModuli) return OZ2_ERR_UNSUPPORTED_R;
  if (k == 0 || !A || !B || !d || !e || !row_flag || !col_flag || !planes_a || !planes_b) return OZ2_ERR_INVALID_ARG;
  DeviceState* ds = nullptr;
  if ((st = device_state(&ds)) != OZ2_OK) return st;
  const Oz2Moduli mods = build_moduli(num_moduli, quant);
  return to_status(launch_deconstruct(m, n, k, mods, ds->table_a, ds->table_b, A, lda, B, ldb, d, e, row_flag, col_flag, quant,
                                      planes_a, planes_b, static_cast<cudaStream_t>(stream)));
}

int oz2_residue_gemm(int64_t m, int64_t n, int64_t k, int num_moduli, const uint8_t* planes_a,
                     const uint8_t* planes_b, int16_t* residues, int64_t ldr, void* stream) {
  if (m <= 0 || n <= 0 || k <= 0 || !planes_a || !planes_b || !residues || ldr < m) return OZ2_ERR_INVALID_ARG;
  if (num_moduli < 1 || num_moduli > kMaxModuli) return OZ2_ERR_UNSUPPORTED_R;
  if (m >= (1LL << 31) || n >= (1LL << 31) || k > (1LL << 24)) return OZ2_ERR_UNSUPPORTED;
  DeviceState* ds = nullptr;
  int st = device_state(&ds);
  if (st) return st;
  const Oz2Moduli mods = build_moduli(num_moduli, OZ2_QUANT_TZ);
  const int64_t k_pad = (k + kKPad - 1) / kKPad * kKPad;
  return to_status(launch_plane_gemm(m, n, k_pad, mods, planes_a, planes_b, 0, residues, ldr, nullptr, ds->status,
                                     static_cast<cudaStream_t>(stream)));
}

int oz2_residue_gemm_simt(int64_t m, int64_t n, int64_t k, int num_moduli, const uint8_t* planes_a,
                          const uint8_t* planes_b, int16_t* residues, int64_t ldr, void* stream) {
  if (m <= 0 || n <= 0 || k <= 0 || !planes_a || !planes_b || !residues || ldr < m) return OZ2_ERR_INVALID_ARG;
  if (num_moduli < 1 || num_moduli > kMaxModuli) return OZ2_ERR_UNSUPPORTED_R;
  DeviceState* ds = nullptr;
  int st = device_state(&ds);
  if (st) return st;
  const Oz2Moduli mods = build_moduli(num_moduli, OZ2_QUANT_TZ);
  const int64_t k_pad = (k + kKPad - 1) / kKPad * kKPad;
  return to_status(launch_plane_gemm(m, n, k_pad, mods, planes_a, planes_b, 2, residues, ldr, nullptr, ds->status,
                                     static_cast<cudaStream_t>(stream)));
}

int oz2_reconstruct(int64_t m, int64_t n, int num_moduli, const int16_t* residues, int64_t ldr, const int32_t* d,
                    const int32_t* e, double* C, int64_t ldc, void* stream) {
  if (m < 0 || n < 0 || ldr < std::max<int64_t>(1, m) || ldc < std::max<int64_t>(1, m)) return OZ2_ERR_INVALID_ARG;
  if (num_moduli < 1 || num_moduli > kMaxModuli) return OZ2_ERR_UNSUPPORTED_R;
  if (m && n && (!residues || !d || !e || !C)) return OZ2_ERR_INVALID_ARG;
  const Oz2Moduli mods = build_moduli(num_moduli, OZ2_QUANT_TZ);
  return to_status(
      launch_reconstruct(m, n, mods, residues, ldr, d, e, C, ldc, static_cast<cudaStream_t>(stream)));
}

int oz2_fallback(int64_t m, int64_t n, int64_t k, const double* A, int64_t lda, const double* B, int64_t ldb,
                 const uint8_t* row_flag, const uint8_t* col_flag, double* C, int64_t ldc, void* stream) {
  int st = check_sizes(m, n, k, lda, ldb, ldc);
  if (st) return st;
  if (m == 0 || n == 0) return OZ2_OK;
  if (!row_flag || !col_flag || !C || (k && (!A || !B))) return OZ2_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int* scratch = nullptr;
  if (pool_alloc(reinterpret_cast<void**>(&scratch), sizeof(int) * (m + n + 2), s) != cudaSuccess) {
    cudaGetLastError();
    return OZ2_ERR_ALLOC;
  }
  cudaError_t err = launch_fallback_lists(m, n, k, A, lda, B, ldb, row_flag, col_flag, scratch, C, ldc, s, true);
  cudaFreeAsync(scratch, s);
  return to_status(err);
}

int oz2_native_dgemm(int64_t m, int64_t n, int64_t k, const double* A, int64_t lda, const double* B, int64_t ldb,
                     double* C, int64_t ldc, void* stream) {
  int st = check_sizes(m, n, k, lda, ldb, ldc);
  if (st) return st;
  if (m == 0 || n == 0) return OZ2_OK;
  if (!C || (k && (!A || !B))) return OZ2_ERR_INVALID_ARG;
  return to_status(launch_native(m, n, k, A, lda, B, ldb, C, ldc, static_cast<cudaStream_t>(stream)));
}

}  // extern "C"
