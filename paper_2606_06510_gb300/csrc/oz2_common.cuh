// Internal definitions shared by the liboz2 translation units.
//
// Modulus constants are computed once per r on the host (oz2_api.cu) and
// passed to kernels by value (__grid_constant__), so concurrent calls with
// different r never share mutable constant memory.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/oz2.h"

namespace oz2 {

constexpr int kMaxModuli = 16;
constexpr int kMaxPlanes = 48;         // 3 per modulus at most
constexpr int kKPad = 128;             // k is padded to a multiple of this
constexpr int kMagClampMax = 9;        // 2^-9: smallest E4M3 magnitude
constexpr int kFallbackWindow = 128;   // binades from the median (fallback)
// Exact FP32 accumulation (Eq. accum-exact), K_slab · max|term| ≤ 2^24:
//  square moduli: terms d0e0 (≤ 256) and d1e0 + d0e1 (≤ 512) → K_slab 32768;
//  nonsquare moduli with the merged accumulator d0e0 - 16·d1e1 (≤ 4095 on
//  the S tail and the extension primes) → K_slab 4096 (4096 · 4095 < 2^24).
constexpr int kKSlabSquare = 32768;
constexpr int kKSlabMerged = 4096;

// The modulus list (§2.5: the published set S in the order the paper lists
// it, then the extension primes for r = 13..16) and per-modulus constants
// derived from it at compile time.
constexpr int kModuliList[kMaxModuli] = {1089, 1024, 961, 841, 625, 529, 511, 509,
                                         503,  499,  491, 487, 479, 467, 463, 461};

// The deconstruction splits each integer entry Ã (|Ã| < 2^62) into 21-bit
// limbs, Ã = v0 + v1·2^21 + v2·2^42 with v0, v1 ∈ [0, 2^21) and v2 signed
// (|v2| ≤ 2^20), and forms per modulus the 32-bit sum
// Y = (v0 + kDecBias) + v1·c1 + v2·c2 ≡ Ã + kDecBias (mod m), with the
// centred limb weights c1 = 2^21 mod m and c2 = 2^42 mod m (|c| ≤ 544).
// kDecBias = 2^31 keeps Y inside (0, 2^32): |v1·c1| < 2^30.1 and
// |v2·c2| < 2^29.1.  The digit-plane table holds 2m entries per nonsquare
// modulus (entry i: the planes of the residue (i - kDecBias) mod m), so that
// a quotient one too large, and the bias, cost nothing at the lookup.
// Square moduli compute their digits.
constexpr uint32_t kDecBias = 1u << 31;
constexpr int kLimbBits = 21;

struct ModConst {
  int m;
  int s;          // square base, 0 for nonsquare moduli
  int plane_off;  // first plane of this modulus
  int table_off;  // nonsquare: first of its 2m entries in the digit-plane table
  int c1, c2;     // centred 2^21 mod m and 2^42 mod m
  uint32_t magic; // ⌈2^32/m⌉
  // Square moduli (digits computed, not looked up): E = (⌊m/2⌋ - kDecBias)
  // mod m, the digit offsets h0 = ⌊s/2⌋ and h1 = ⌈(⌊m/2⌋ - h0)/s⌉, and
  // ⌈2^17/s⌉ (⌊u·⌈2^17/s⌉/2^17⌋ = ⌊u/s⌋ for u < 2^17/s).
  uint32_t sq_e;
  int sq_h0, sq_h1;
  int sq_c17;
};

// x mod m in [-⌊m/2⌋, m - 1 - ⌊m/2⌋] (the centred residue) for x ≥ 0.
constexpr int ce_centred(unsigned long long x, int m) {
  const int r = static_cast<int>(x % static_cast<unsigned long long>(m));
  return r > m - 1 - m / 2 ? r - m : r;
}

constexpr int ce_isqrt(int m) {
  int s = 0;
  while ((s + 1) * (s + 1) <= m) ++s;
  return s * s == m ? s : 0;
}
// Digit planes of an operand with `rows` rows are stored as 128 × 128-byte
// blocks: rows are padded to a multiple of 128 (the pad rows hold zero
// digits), and byte l of row `row` of plane p is at
//   ((⌊row/128⌋·(k_pad/128) + ⌊l/128⌋)·P + p)·2^14 + (row mod 128)·128 + l mod 128
// for P planes in all.  One block is exactly the tile the residue GEMM loads
// for an MMA operand (one contiguous 16 KiB TMA box), and the P blocks of a
// (row block, k-block) are consecutive, so a thread of the deconstruction
// reaches the same row segment of every plane at compile-time offsets.
constexpr int kPlaneLine = 128;                            // bytes of a row segment (k-entries)
constexpr int kPlaneRows = 128;                            // rows of a block
constexpr int kPlaneBlock = kPlaneLine * kPlaneRows;       // 16 KiB

// Planes stored for the first r moduli (two per square modulus, three per
// nonsquare one).
constexpr int num_planes(int r) {
  int p = 0;
  for (int j = 0; j < r; ++j) p += ce_isqrt(kModuliList[j]) ? 2 : 3;
  return p;
}

constexpr ModConst mod_const(int i) {
  ModConst c{};
  int plane = 0, toff = 0;
  for (int j = 0; j < i; ++j) {
    plane += ce_isqrt(kModuliList[j]) ? 2 : 3;
    toff += ce_isqrt(kModuliList[j]) ? 0 : kModuliList[j];  // the table holds nonsquare moduli only
  }
  const int m = kModuliList[i];
  c.m = m;
  c.s = ce_isqrt(m);
  c.plane_off = plane;
  c.table_off = 2 * toff;
  const unsigned long long um = static_cast<unsigned long long>(m);
  c.c1 = ce_centred(1ull << kLimbBits, m);
  c.c2 = ce_centred(1ull << (2 * kLimbBits), m);
  c.magic = static_cast<uint32_t>(((1ull << 32) + um - 1) / um);
  if (c.s) {
    const int H = m / 2;
    c.sq_e = static_cast<uint32_t>((static_cast<long long>(H) - kDecBias % um + m) % m);
    c.sq_h0 = c.s / 2;
    c.sq_h1 = (H - c.sq_h0 + c.s - 1) / c.s;
    c.sq_c17 = ((1 << 17) + c.s - 1) / c.s;
  }
  return c;
}

// Device status word values (stored in Oz2Device::status).
constexpr int kStatusTimeout = 1;

struct Oz2Moduli {
  int r;
  int nplanes;
  int T;                        // range exponent of the scale choice
  int m[kMaxModuli];
  int sq_base[kMaxModuli];      // s for m = s², 0 for nonsquare
  int plane_off[kMaxModuli];    // first plane of modulus i
  // Garner (Eq. garner): pmod[k][j] = (m_0 ⋯ m_{j-1}) mod m_k for j < k,
  // inv[k] = (m_0 ⋯ m_{k-1})^-1 mod m_k, goff[k] = multiple of m_k ≥ 2^27.
  int pmod[kMaxModuli][kMaxModuli];
  int inv[kMaxModuli];
  uint32_t invp[kMaxModuli];    // ⌊inv[k]·2^32 / m_k⌋ (Shoup's precomputed quotient)
  int goff[kMaxModuli];
  // M and ⌈M/2⌉ as 3×64-bit little-endian limbs.
  unsigned long long M[3];
  unsigned long long Mhalf[3];
  // Direct CRT (fast path of the reconstruction): W_k = (M/m_k)·y_k with
  // y_k = (M/m_k)^-1 mod m_k as 32-bit limbs, F_k = round(2^32·y_k/m_k), and
  // coff_k = m_k·⌈2^15/m_k⌉ (makes any int16 residue nonnegative).
  uint32_t crtw[kMaxModuli][5];
  uint32_t crtf[kMaxModuli];
  int coff[kMaxModuli];
  // Two-word direct CRT (r ≤ 12, M < 2^112), for signed 32×32→64-bit
  // multiply-adds: F_k = round(2^64·y_k/m_k) mod 2^64 = fh·2^32 + fl and
  // W_k mod 2^64 = wh·2^32 + wl, each with a signed low word;
  // g_k = round(2^18·y_k/m_k); M mod 2^64 = mlh·2^32 + ml and
  // round(M/2^51) = m51h·2^32 + m51l (ml, m51l signed).
  int crt_fl[kMaxModuli], crt_fh[kMaxModuli];
  int crt_wl[kMaxModuli], crt_wh[kMaxModuli];
  int crt_g[kMaxModuli];
  int crt_ml, crt_mlh;
  int crt_m51l, crt_m51h;
  // 96-bit direct CRT of the fused kernel (r = 11, 12): F_k = round(2^96·y_k/m_k)
  // = y2·2^64 + y1·2^32 + y0 with y0 and y1 signed low words; M as four
  // 32-bit words; and a bound on |X| - ⌊|Y|·M/2^96⌋ for centred residues.
  int crt_y0[kMaxModuli], crt_y1[kMaxModuli];
  uint32_t crt_y2[kMaxModuli];
  uint32_t crt_m32[4];
  unsigned long long crt_err_centred;
  int table_entries;            // 2·Σ m_i over the nonsquare moduli (digit-plane table)
};

// Per-device status block (in device global memory, owned by oz2_api.cu).
struct Oz2Device {
  int status;                   // 0, or kStatusTimeout (sticky until read)
  int timeout_site;
  int fallback_rows;
  int fallback_cols;
  int u_max_bits;               // float bits of max_ij U_ij ("+1" pass)
  int s;                        // column budget (R2) or pB (R1)
  int pad[10];
};


// ---------------------------------------------------------------------------
// PTX wrappers (sm_100-family tcgen05 / TMA / mbarrier), with bounded waits.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count));
}

__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n"
      " mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait for the given phase parity; gives up after ~`limit` clock cycles and
// returns false.  Every spin in the library goes through this.
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity, long long limit) {
  if (mbar_try_wait(bar, parity)) return true;
  long long t0 = clock64();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 255u) == 0 && clock64() - t0 > limit) return false;
  }
}

// 3-D tiled TMA load into shared memory, completing on an mbarrier.
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, uint32_t bar,
                                           int x, int y, int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(x), "r"(y), "r"(z)
      : "memory");
}

// 2-D tiled TMA load into this CTA's shared memory, completing on an mbarrier.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint32_t bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(x), "r"(y)
      : "memory");
}

__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// --- clusters (CTA pairs) ----------------------------------------------------
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// shared::cluster address of the same shared-memory offset in CTA `rank`.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Arrive on an mbarrier of another CTA of the cluster (address from mapa_shared).
__device__ __forceinline__ void mbar_arrive_remote(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}
// The same arrive without release semantics: it orders none of the thread's
// earlier memory operations (a release would hold the arrive until the
// thread's outstanding global stores are performed).  For a thread whose
// tensor-memory loads have completed (tcgen05.wait::ld, then
// tcgen05.fence::before_thread_sync), program order alone puts those loads
// before the arrive.
__device__ __forceinline__ void mbar_arrive_remote_relaxed(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}
// 3-D tiled TMA load issued by either CTA of a pair; the transaction bytes
// complete on `bar` (a shared::cluster address, here the leader CTA's barrier).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* map, uint32_t bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cta.global.tile.mbarrier::complete_tx::bytes.cta_group::2"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(x), "r"(y)
      : "memory");
}
__device__ __forceinline__ void tma_load_3d_pair(uint32_t dst, const CUtensorMap* map, uint32_t bar, int x, int y,
                                                 int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cta.global.tile.mbarrier::complete_tx::bytes.cta_group::2"
      " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(x), "r"(y), "r"(z)
      : "memory");
}

// --- tcgen05, CTA pair (cta_group::2) -------------------------------------------
__device__ __forceinline__ void tmem_alloc_pair(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
// D[tmem] (+)= A·Bᵀ over the CTA pair (M = 256: 128 rows of A in each CTA's
// shared memory at the same offset; B split likewise), issued by the leader.
__device__ __forceinline__ void mma_f8_pair(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::2.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive once on the barrier at this shared offset in every CTA of `mask`
// when all prior tcgen05 ops of the issuing thread complete.
__device__ __forceinline__ void mma_commit_pair_mc(uint32_t bar, uint16_t mask) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
          bar),
      "h"(mask)
      : "memory");
}
__device__ __forceinline__ void mma_commit_pair(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}

// --- tcgen05 -----------------------------------------------------------------
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem] · B[smem]^T, kind::f8f6f4, issued by one thread.
__device__ __forceinline__ void mma_f8(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                       uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive on an mbarrier once all prior tcgen05 ops of this thread complete.
__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
      : "memory");
}

// 32 lanes × 32 bits, 32 consecutive columns per thread.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
        "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
        "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]),
        "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]), "=r"(v[25]),
        "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr));
}
// 32 lanes × 32 bits, 4 consecutive columns per thread.
__device__ __forceinline__ void tmem_ld4(uint32_t taddr, uint32_t (&v)[4]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3])
               : "r"(taddr));
}
// 32 lanes × 32 bits, 4 consecutive columns per thread, stored.
__device__ __forceinline__ void tmem_st4(uint32_t taddr, const uint32_t (&v)[4]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x4.b32 [%0], {%1,%2,%3,%4};" ::"r"(taddr), "r"(v[0]), "r"(v[1]),
               "r"(v[2]), "r"(v[3])
               : "memory");
}
// 32 lanes × 32 bits, 8 consecutive columns per thread.
__device__ __forceinline__ void tmem_ld8(uint32_t taddr, uint32_t (&v)[8]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
               : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7])
               : "r"(taddr));
}
// 32 lanes × 32 bits, 16 consecutive columns per thread.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&v)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
        "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
      : "r"(taddr));
}
// 32 lanes × 32 bits, 16 consecutive columns per thread, stored.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&v)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]),
      "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
      : "memory");
}
__device__ __forceinline__ void tmem_st_wait() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_ld_wait() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor for a K-major operand tile stored with the
// 128-byte swizzle that TMA writes (rows of 128 bytes, 8-row atoms of 1024
// bytes): start address >> 4 in bits [0,14), leading-byte offset (unused for
// swizzled K-major, set to 1) in [16,30), stride-byte offset 1024 >> 4 in
// [32,46), descriptor version 1 in [46,48), layout SWIZZLE_128B (2) in [61,64).
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);
  d |= static_cast<uint64_t>(1u) << 16;
  d |= static_cast<uint64_t>(1024u >> 4) << 32;
  d |= static_cast<uint64_t>(1u) << 46;
  d |= static_cast<uint64_t>(2u) << 61;
  return d;
}

// Shared-memory matrix descriptor for a K-major operand tile without
// swizzle: 8-row × 16-byte core matrices, each stored as 128 contiguous
// bytes; `lbo` is the byte distance between core matrices adjacent in K and
// `sbo` between core matrices adjacent in M (or N).  Start address >> 4 in
// bits [0,14), LBO >> 4 in [16,30), SBO >> 4 in [32,46), descriptor version
// 1 in [46,48), layout SWIZZLE_NONE (0) in [61,64).
__device__ __forceinline__ uint64_t smem_desc_plain(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32;
  d |= static_cast<uint64_t>(1u) << 46;
  return d;
}

// Instruction descriptor, kind::f8f6f4: D = F32 (bits 4-5 = 1), A = B = E4M3
// (bits 7-9, 10-12 = 0), both K-major (bits 15, 16 = 0), N >> 3 in bits
// 17-22, M >> 4 in bits 24-28.
__host__ __device__ constexpr uint32_t idesc_f8_f32(int M, int N) {
  return (1u << 4) | (static_cast<uint32_t>(N >> 3) << 17) | (static_cast<uint32_t>(M >> 4) << 24);
}

}  // namespace oz2

// Host-side launchers (defined in the kernel translation units).
namespace oz2 {
// Counts kernel launches made by the library (read through oz2_get_stats).
void count_launch(int n = 1);

// Programmatic dependent launch: the kernel may be scheduled while the
// kernel before it in the stream is still running (once every block of that
// one has called pdl_trigger() or exited), so its launch latency overlaps
// the predecessor's tail.  It must call pdl_wait(), which returns once the
// predecessor has completed and its writes are visible, before it reads
// anything the predecessor wrote.  Launched the ordinary way, pdl_wait()
// returns at once.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_dependent(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                                   Args... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
struct ScanOut {
  int32_t* ra;
  int32_t* cb;
  uint8_t* row_flag;
  uint8_t* col_flag;
};
cudaError_t launch_scan(int64_t m, int64_t n, int64_t k, const double* A, int64_t lda,
                        const double* B, int64_t ldb, unsigned flags, ScanOut out,
                        Oz2Device* dev, cudaStream_t st, bool zero_keys);
cudaError_t launch_magnitude_planes(int64_t m, int64_t n, int64_t k, const double* A,
                                    int64_t lda, const double* B, int64_t ldb, const int32_t* ra,
                                    const int32_t* cb, const uint8_t* row_flag,
                                    const uint8_t* col_flag, uint8_t* mag_a, uint8_t* mag_b,
                                    cudaStream_t st);
cudaError_t launch_choose_scales(int64_t m, int64_t n, int64_t k, const Oz2Moduli& mods,
                                 int scale_mode, const float* urow, const int32_t* ra,
                                 const int32_t* cb, const uint8_t* row_flag,
                                 const uint8_t* col_flag, int32_t* d, int32_t* e,
                                 Oz2Device* dev, cudaStream_t st);
cudaError_t launch_deconstruct(int64_t m, int64_t n, int64_t k, const Oz2Moduli& mods,
                               const uint32_t* table_a, const uint32_t* table_b,
                               const double* A, int64_t lda,
                               const double* B, int64_t ldb, const int32_t* d, const int32_t* e,
                               const uint8_t* row_flag, const uint8_t* col_flag, int quant,
                               uint8_t* planes_a, uint8_t* planes_b, cudaStream_t st);
// Parts of K per unit the residue GEMM takes for an m×n C (1: no split),
// with the r moduli of which the first nsq are squares, residues with
// leading dimension ldr, partial_bytes of scratch and `pairs` CTA pairs.
// Host-only arithmetic.
int64_t residue_gemm_kparts(int64_t m, int64_t n, int64_t k_pad, int r, int nsq, int64_t ldr, size_t partial_bytes,
                            int64_t pairs);
int64_t magnitude_gemm_kparts(int64_t m, int64_t n, int64_t k_pad, size_t scratch_bytes, int64_t pairs);
// `partials` (16-byte aligned, `partial_bytes` long, or null) is scratch the
// residue GEMM may split K into (the parts' residues), and the magnitude GEMM
// too (the m×n FP32 sums of its parts); it must not overlap the operands,
// C^(i) or urow.
cudaError_t launch_plane_gemm(int64_t m, int64_t n, int64_t k_pad, const Oz2Moduli& mods,
                              const uint8_t* planes_a, const uint8_t* planes_b, int mode,
                              int16_t* residues, int64_t ldr, float* urow, Oz2Device* dev, cudaStream_t st,
                              int16_t* partials = nullptr, size_t partial_bytes = 0);
// `centred`: every residue lies in [-⌊m_k/2⌋, m_k-1-⌊m_k/2⌋] (as the residue
// GEMM writes them); otherwise any int16 representative.
cudaError_t launch_reconstruct(int64_t m, int64_t n, const Oz2Moduli& mods,
                               const int16_t* residues, int64_t ldr, const int32_t* d,
                               const int32_t* e, double* C, int64_t ldc, cudaStream_t st);
cudaError_t launch_fallback_lists(int64_t m, int64_t n, int64_t k, const double* A, int64_t lda,
                                  const double* B, int64_t ldb, const uint8_t* row_flag,
                                  const uint8_t* col_flag, int* scratch, double* C, int64_t ldc,
                                  cudaStream_t st, bool zero_counts);
// The tensor-pipe rate probe (k_gemm.cu); reports the CTA pairs it runs on.
cudaError_t launch_mma_rate(int64_t iters, Oz2Device* dev, int* pairs_out, cudaStream_t st);
// The fused residue GEMM and reconstruction (k_fused.cu) for r = 11, 12 and
// k_pad ≤ kFusedMaxKPad: C from the digit planes, without residue matrices.
// `scratch` (scratch_bytes, 16-byte aligned, at least 16 + 8·m·n bytes)
// holds the list of outputs the fast reconstruction leaves.
constexpr int64_t kFusedMaxKPad = 256;
bool fused_crt_applies(int64_t k_pad, int r);
cudaError_t launch_fused_crt(int64_t m, int64_t n, int64_t k_pad, const Oz2Moduli& mods, const uint8_t* planes_a,
                             const uint8_t* planes_b, const int32_t* d, const int32_t* e, const uint8_t* row_flag,
                             const uint8_t* col_flag, double* C, int64_t ldc, void* scratch, size_t scratch_bytes,
                             Oz2Device* dev, cudaStream_t st);
// On-the-fly residues (k_deconstruct.cu): the residue GEMM of a skinny C
// (n ≤ kModeFMaxN) with A's digit planes formed in shared memory from A
// itself, never stored; B's planes come from the deconstruction.  Writes the
// residue matrices as the residue GEMM does.
constexpr int64_t kModeFMaxN = 32;
bool modef_applies(int64_t m, int64_t n, int64_t k_pad);
cudaError_t launch_modef(int64_t m, int64_t n, int64_t k, const Oz2Moduli& mods, const uint32_t* table_a,
                         const double* A, int64_t lda, const int32_t* d, const uint8_t* row_flag, int quant,
                         const uint8_t* planes_b, int16_t* residues, int64_t ldr, Oz2Device* dev, cudaStream_t st);
cudaError_t launch_native(int64_t m, int64_t n, int64_t k, const double* A, int64_t lda,
                          const double* B, int64_t ldb, double* C, int64_t ldc, cudaStream_t st);
}  // namespace oz2
