// Phase 2 of Ozaki Scheme II on FP8 tensor cores (§2.3 Eq. modgemm; §2.5
// Eq. sq-shortcut, Eq. kar, Eq. accum-exact) and the "+1" magnitude GEMM of
// §2.4, as one persistent tcgen05 kernel for sm_103a running on CTA pairs.
//
// Work unit = (modulus, 256×256 output tile); units are taken modulus-major
// so that the planes of one modulus stay in L2 while every pair works on it.
// The nonsquare moduli, whose units load three stage pairs per k-block
// against two for a square modulus, come first, and successive waves of
// units are dealt to the pairs in alternating directions, so that the pairs
// that take a heavy unit in one wave take a light one in the next.
// A pair (cluster of 2 CTAs) computes its tile with cta_group::2 MMAs of
// M = N = 256, K = 32: each CTA holds 128 rows of the A plane tile and 128
// rows of the B plane tile in its own shared memory, and 128 rows × 256
// columns of each FP32 accumulator in its tensor memory.
//
// Per modulus the three plane products of §2.5 accumulate into two TMEM
// accumulators (256 columns each):
//   square m = s²  : acc0 += d0·e0,            acc1 += d1·e0 + d0·e1
//   nonsquare m    : acc0 += (d0+d1)(e0+e1),   acc1 += d0·e0 + (-16 d1)·e1
// (the A operand stores its last nonsquare plane pre-scaled by -2^b, the
// accumulator merge of §2.5 "Accumulators").  Every K-slab (32768 squares,
// 4096 nonsquare: Eq. accum-exact) the epilogue reads the accumulators and
// forms  v = acc0 + s·acc1  or  v = 16·acc0 - 15·acc1  mod m.  After a slab
// that is not the last it writes the centred residue back into the
// accumulators (tcgen05.st) for the next slab to accumulate on; after the
// last it stores the centred residue as int16, column-major (each thread
// owns one row; a warp's store covers 32 consecutive rows of one column, 64
// contiguous bytes).
//
// Pipeline: a stage is one (A plane, B plane) pair of 128-byte-deep tiles
// (32 KiB per CTA), six stages.  Warp 0 of each CTA issues its CTA's TMA
// loads, completing on the leader's stage barrier; warp 1 of the leader
// issues the MMAs and multicasts stage releases and accumulator-ready
// signals to both CTAs; warps 2..17 of both CTAs run the epilogue (64
// columns each) and release the accumulators to the leader.  Every wait is bounded; on expiry the
// kernel records OZ2_ERR_TIMEOUT in the device status word and drains.
#include <algorithm>

#include "oz2_gemm.cuh"

namespace oz2 {

constexpr int kTileM = 256, kTileN = 256;        // per CTA pair
constexpr int kStageBytes = 2 * kTileBytes;      // A tile + B tile
constexpr int kStages = 6;
constexpr int kEpiWarps = 16;
constexpr int kGemmThreads = 32 * (2 + kEpiWarps);  // producer, MMA, epilogue
constexpr int kTmemCols = 512;
constexpr int kAccCols = 256;
constexpr int kGroupM = 8;                       // tile rasterisation group

struct EpiCtx {
  int16_t* res;   // r × (m×n column-major, ld = ldr ≥ m; matrix i at i·n·ldr)
  float* urow;
  Oz2Device* dev;
  int64_t m, n, ldr;
  float* upart;   // magnitude GEMM split along k: U (m×n row-major, ld = ldu) summed over the parts
  int64_t ldu;    // a multiple of 4: 16-byte rows
};

// Units: (modulus, part of the k-blocks, tile).  With kparts > 1 (split K)
// each unit covers kpart_steps consecutive k-blocks (the last part fewer)
// and the epilogue stores its residue as part `part` of the partial-residue
// planes, which fold_parts_kernel then sums mod m (Eq. modgemm is a sum over
// k, so C^(i) is the sum of the parts' residues mod m_i).
struct UnitMap {
  int64_t ntm, ntn, ntiles, nunits;
  int nsq, nheavy;  // leading square moduli; nonsquare moduli after them
  int64_t ksteps, kparts, kpart_steps;
};

struct Unit {
  int i, part;         // modulus, part of the k-blocks
  int64_t tm, tn;      // tile
  int64_t k_lo, k_hi;  // k-blocks [k_lo, k_hi)
};

// Unit u (grouped raster of kGroupM tile rows).  Modulus block j of the
// units is modulus nsq + j for the nheavy nonsquare moduli, then modulus
// j - nheavy for the squares; within a modulus the parts come in order.
// The magnitude GEMM (MODE 1) has one modulus; its parts of k (when it is
// split) come in order, each over all tiles.
template <int MODE>
__device__ __forceinline__ Unit unit_at(int64_t u, const UnitMap& um) {
  Unit x;
  int64_t t = u;
  if (MODE == 1) {
    x.i = 0;
    x.part = static_cast<int>(u / um.ntiles);
    t = u - static_cast<int64_t>(x.part) * um.ntiles;
  } else {
    const int64_t per_mod = um.ntiles * um.kparts;
    const int j = static_cast<int>(u / per_mod);
    x.i = j < um.nheavy ? um.nsq + j : j - um.nheavy;
    const int64_t v = u - static_cast<int64_t>(j) * per_mod;
    x.part = static_cast<int>(v / um.ntiles);
    t = v - static_cast<int64_t>(x.part) * um.ntiles;
  }
  const int64_t per_group = kGroupM * um.ntn;
  const int64_t g = t / per_group;
  const int64_t first = g * kGroupM;
  const int64_t gm = um.ntm - first < kGroupM ? um.ntm - first : kGroupM;
  const int64_t local = t - g * per_group;
  x.tm = first + local % gm;
  x.tn = local / gm;
  x.k_lo = static_cast<int64_t>(x.part) * um.kpart_steps;
  x.k_hi = um.ksteps - x.k_lo < um.kpart_steps ? um.ksteps : x.k_lo + um.kpart_steps;
  return x;
}

// The unit a pair takes in wave w: waves of npairs units, dealt to the pairs
// in ascending order in even waves and descending order in odd ones.
__device__ __forceinline__ int64_t wave_unit(int64_t pair, int64_t w, int64_t npairs) {
  return w * npairs + ((w & 1) ? npairs - 1 - pair : pair);
}

template <int MODE>
__device__ __forceinline__ int planes_of(const Oz2Moduli& mods, int i) {
  return MODE == 0 ? (mods.sq_base[i] ? 2 : 3) : 1;
}
template <int MODE>
__device__ __forceinline__ int64_t slab_steps_of(const Oz2Moduli& mods, int i, int64_t ksteps) {
  if (MODE == 1) return ksteps;  // the magnitude sums stay below 2^24 units over all of k
  return (mods.sq_base[i] ? kKSlabSquare : kKSlabMerged) / kBK;
}

// MODE 0: residue planes (all moduli); MODE 1: magnitude planes ("+1" pass).
// SHORT1, for MODE 0: the instance for k ≤ 128 (one k-block, so one short
// slab for every modulus), whose epilogue takes the single-correction
// reduction; for MODE 1: the instance whose tiles run in parts of k and add
// their partial sums into U (EpiCtx::upart) instead of taking row maxima.
template <int MODE, bool SHORT1 = false>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kGemmThreads, 1)
    plane_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                      const __grid_constant__ Oz2Moduli mods, int64_t k_pad, UnitMap um, EpiCtx ctx) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
  // bars: full[S], empty[S], acc_full, acc_empty, drain
  __shared__ uint32_t tmem_base_s;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int64_t pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
  const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + kStages);
  const uint32_t acc_full = smem_u32(bars + 2 * kStages), acc_empty = smem_u32(bars + 2 * kStages + 1);
  const uint32_t drain_bar = smem_u32(bars + 2 * kStages + 2);
  const int64_t ksteps = k_pad / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, 2 * kEpiWarps);
    mbar_init(drain_bar, 1);
    fence_barrier_init();
    prefetch_tensormap(&tmA);
    prefetch_tensormap(&tmB);
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(&tmem_base_s), kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  bool ok = true;

  if (warp == 0) {
    // ---------------- TMA producer (both CTAs) ----------------
    if (lane == 0) {
      uint32_t it = 0;
      const uint32_t full_leader0 = mapa_shared(full0, 0);
      for (int64_t w = 0, u = pair; u < um.nunits && ok; u = wave_unit(pair, ++w, npairs)) {
        const Unit x = unit_at<MODE>(u, um);
        const int i = x.i;
        const int64_t tm = x.tm, tn = x.tn;
        const int np = planes_of<MODE>(mods, i);
        const int pbase = MODE == 0 ? mods.plane_off[i] : 0;
        const int ya = static_cast<int>(tm * kTileM + rank * kRows);
        const int yb = static_cast<int>(tn * kTileN + rank * kRows);
        // Digit planes: first line of block (row block, k-block 0, plane pbase);
        // successive k-blocks are nplanes blocks apart.  A row block past the
        // operand's last one lies past the end of the tensor (zero fill).
        const int64_t blk_a = (static_cast<int64_t>(ya / kPlaneRows) * ksteps * mods.nplanes + pbase) * kPlaneRows;
        const int64_t blk_b = (static_cast<int64_t>(yb / kPlaneRows) * ksteps * mods.nplanes + pbase) * kPlaneRows;
        for (int64_t kb = x.k_lo; kb < x.k_hi && ok; ++kb) {
          for (int p = 0; p < np; ++p, ++it) {
            const int s = it % kStages;
            if (!mbar_wait_bounded(empty0 + 8 * s, ((it / kStages) & 1) ^ 1, kWaitLimit)) {
              ok = false;
              break;
            }
            if (leader) mbar_arrive_expect_tx(full0 + 8 * s, 2u * kStageBytes);
            const uint32_t sa = smem_u32(smem + s * kStageBytes);
            if (MODE == 0) {
              const int64_t off = (kb * mods.nplanes + p) * kPlaneRows;
              tma_load_2d_pair(sa, &tmA, full_leader0 + 8 * s, 0, static_cast<int>(blk_a + off));
              tma_load_2d_pair(sa + kTileBytes, &tmB, full_leader0 + 8 * s, 0, static_cast<int>(blk_b + off));
            } else {
              const int x = static_cast<int>(kb * kBK);
              tma_load_3d_pair(sa, &tmA, full_leader0 + 8 * s, x, ya, 0);
              tma_load_3d_pair(sa + kTileBytes, &tmB, full_leader0 + 8 * s, x, yb, 0);
            }
          }
        }
      }
      if (!ok) {
        ctx.dev->status = kStatusTimeout;
        ctx.dev->timeout_site = 1;
      }
      if (leader)  // the leader's stage barriers also count the peer's bytes
        for (uint32_t j = (it > kStages ? it - kStages : 0); j < it; ++j)
          mbar_wait_bounded(full0 + 8 * (j % kStages), (j / kStages) & 1, kWaitLimit);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer (leader CTA) ----------------
    if (leader && lane == 0) {
      constexpr uint32_t idesc = idesc_f8_f32(kTileM, kTileN);
      // Stage s, operand o, k-chunk kk: the descriptor of stage 0 plus the
      // byte offset >> 4 (the start-address field has room: smem < 256 KiB).
      const uint64_t desc0 = smem_desc_sw128(smem_u32(smem));
      uint32_t st = 0, ph = 0, accph = 0;   // current stage and its full-barrier parity
      auto next = [&](uint32_t& s_, uint32_t& p_) {
        if (++s_ == kStages) {
          s_ = 0;
          p_ ^= 1;
        }
      };
      for (int64_t w = 0, u = pair; u < um.nunits && ok; u = wave_unit(pair, ++w, npairs)) {
        const Unit x = unit_at<MODE>(u, um);
        const int i = x.i;
        const int np = planes_of<MODE>(mods, i);
        const int64_t slab = slab_steps_of<MODE>(mods, i, ksteps);
        for (int64_t kb0 = x.k_lo; kb0 < x.k_hi && ok; kb0 += slab) {
          if (!mbar_wait_bounded(acc_empty, accph ^ 1, kWaitLimit)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const int64_t kb1 = min(x.k_hi, kb0 + slab);
          for (int64_t kb = kb0; kb < kb1 && ok; ++kb) {
            const uint32_t first = kb == x.k_lo ? 0u : 1u;  // later slabs add to the carried residue
            if (np == 2) {  // square: stages (d0,e0) and (d1,e1)
              uint32_t s1 = st, p1 = ph;
              next(s1, p1);
              if (!mbar_wait_bounded(full0 + 8 * st, ph, kWaitLimit) || !mbar_wait_bounded(full0 + 8 * s1, p1, kWaitLimit)) {
                ok = false;
                break;
              }
              tc_fence_after();
              const uint64_t a0 = desc0 + st * (kStageBytes >> 4), b0 = a0 + (kTileBytes >> 4);
              const uint64_t a1 = desc0 + s1 * (kStageBytes >> 4), b1 = a1 + (kTileBytes >> 4);
#pragma unroll
              for (int kk = 0; kk < kBK / 32; ++kk) {
                const uint32_t acc = kk ? 1u : first;
                mma_f8_pair(tmem, a0 + 2 * kk, b0 + 2 * kk, idesc, acc);                 // d0·e0
                mma_f8_pair(tmem + kAccCols, a1 + 2 * kk, b0 + 2 * kk, idesc, acc);      // d1·e0
                mma_f8_pair(tmem + kAccCols, a0 + 2 * kk, b1 + 2 * kk, idesc, 1u);       // + d0·e1
              }
              mma_commit_pair_mc(empty0 + 8 * st, 0x3);
              mma_commit_pair_mc(empty0 + 8 * s1, 0x3);
              st = s1;
              ph = p1;
              next(st, ph);
            } else {
              for (int p = 0; p < np; ++p) {  // nonsquare: Σ·Σ → acc0; d0e0, -16 d1·e1 → acc1
                if (!mbar_wait_bounded(full0 + 8 * st, ph, kWaitLimit)) {
                  ok = false;
                  break;
                }
                tc_fence_after();
                const uint32_t col = p == 0 ? 0u : kAccCols;
                const uint64_t a = desc0 + st * (kStageBytes >> 4), b = a + (kTileBytes >> 4);
#pragma unroll
                for (int kk = 0; kk < kBK / 32; ++kk) {
                  const uint32_t acc = (kk || p == 2) ? 1u : first;
                  mma_f8_pair(tmem + col, a + 2 * kk, b + 2 * kk, idesc, acc);
                }
                mma_commit_pair_mc(empty0 + 8 * st, 0x3);
                next(st, ph);
              }
            }
          }
          if (!ok) break;
          mma_commit_pair_mc(acc_full, 0x3);  // accumulators complete for this slab, both CTAs
          accph ^= 1;
        }
      }
      if (!ok) {
        ctx.dev->status = kStatusTimeout;
        ctx.dev->timeout_site = 2;
      }
      // All MMAs retired before the tensor memory or the peer's shared memory goes away.
      mma_commit_pair(drain_bar);
      mbar_wait_bounded(drain_bar, 0, kWaitLimit);
    }
    __syncwarp();
  } else {
    // ---------------- epilogue (warps 2..17, both CTAs) ----------------
    const int q = warp & 3;                    // TMEM lane quarter of this warp
    const int h = (warp - 2) >> 2;             // 64-column quarter of the tile
    const uint32_t lane_addr = tmem + (static_cast<uint32_t>(32 * q) << 16) + static_cast<uint32_t>(64 * h);
    const uint32_t acc_empty_leader = mapa_shared(acc_empty, 0);
    uint32_t accph = 0;
    for (int64_t w = 0, u = pair; u < um.nunits && ok; u = wave_unit(pair, ++w, npairs)) {
      const Unit x = unit_at<MODE>(u, um);
      const int i = x.i;
      const int64_t tm = x.tm, tn = x.tn;
      const int64_t row = tm * kTileM + rank * kRows + 32 * q + lane;
      const int64_t col0 = tn * kTileN + 64 * h;
      const bool square = MODE == 0 ? mods.sq_base[i] != 0 : true;
      const float mf = MODE == 0 ? static_cast<float>(mods.m[i]) : 1.f;
      const float inv = 1.f / mf;
      const float sb = MODE == 0 ? static_cast<float>(mods.sq_base[i]) : 0.f;
      const float hi = MODE == 0 ? static_cast<float>(mods.m[i] - 1 - mods.m[i] / 2) : 0.f;
      // This thread's row of C^(i) (of part `part` of it under split K);
      // column j at rrow[j·ldr] (a warp stores 32 consecutive rows of one
      // column, 64 contiguous bytes, per instruction).
      int16_t* rrow =
          MODE == 0 ? ctx.res + (static_cast<size_t>(x.part) * mods.r + i) * ctx.n * ctx.ldr + row : nullptr;
      const int64_t slab = slab_steps_of<MODE>(mods, i, ksteps);
      // Short slabs (K = 128·(k_hi - k_lo) k-entries): v stays an integer below 2^24
      // without reducing the accumulators first.  Square moduli (|d0e0| ≤ 256,
      // |d1e0 + d0e1| ≤ 512, s ≤ 33): |v| ≤ K(256 + 33·512) < 2^24 for K ≤ 896.
      // Nonsquare (|(d0+d1)(e0+e1)| ≤ 22², merged term ≤ 4095):
      // |16·acc0 - 15·acc1| ≤ K(16·484 + 15·4095) < 2^24 for K ≤ 128.
      const bool short_slab = MODE == 0 && x.k_hi - x.k_lo <= (square ? 7 : 1);
      float rowmax = 0.f;
      for (int64_t kb0 = x.k_lo; kb0 < x.k_hi; kb0 += slab) {
        if (!mbar_wait_bounded(acc_full, accph, kWaitLimit)) {
          ok = false;
          break;
        }
        tc_fence_after();
        // A slab other than the last leaves its centred residue r in the
        // accumulators and the next slab accumulates on top of it: acc0 = r,
        // acc1 = 0 for square moduli (v = acc0 + s·acc1), and acc0 = acc1 = r
        // for nonsquare ones (16r - 15r = r).  The bounds of Eq. accum-exact
        // keep their margin: 32768·256 + 544 and 4096·4095 + 255 < 2^24.
        const bool carry = MODE == 0 && kb0 + slab < x.k_hi;
        for (int c = 0; c < 64; c += 16) {
          uint32_t v0[16], v1[16];
          tmem_ld16(lane_addr + c, v0);
          if (MODE == 0) tmem_ld16(lane_addr + kAccCols + c, v1);
          tmem_ld_wait();
          if (c == 48 && !carry) {
            // The last chunk is in registers: release the accumulators now,
            // so the next unit's MMAs overlap this chunk's reduction and
            // stores.  The arrive is relaxed: the residue stores before it
            // need no ordering against the MMAs, and a release would wait
            // for them to be performed.
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_remote_relaxed(acc_empty_leader);
          }
          if (MODE == 1 && SHORT1) {  // a part of k: add this tile's partial sums into U
            const int64_t cc = col0 + c;
            if (row < ctx.m) {
              float* dst = ctx.upart + row * ctx.ldu + cc;  // 16-byte aligned: ldu and cc multiples of 4
              if (cc + 16 <= ctx.n) {
#pragma unroll
                for (int j = 0; j < 16; j += 4)
                  atomicAdd(reinterpret_cast<float4*>(dst + j),
                            make_float4(__uint_as_float(v0[j]), __uint_as_float(v0[j + 1]), __uint_as_float(v0[j + 2]),
                                        __uint_as_float(v0[j + 3])));
              } else {
#pragma unroll
                for (int j = 0; j < 16; ++j)
                  if (cc + j < ctx.n) atomicAdd(dst + j, __uint_as_float(v0[j]));
              }
            }
          } else if (MODE == 1) {
#pragma unroll
            for (int j = 0; j < 16; ++j) rowmax = fmaxf(rowmax, __uint_as_float(v0[j]));
          } else if (carry) {  // every lane: tcgen05.st is warp-collective
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const float rj =
                  combine_residue(__uint_as_float(v0[j]), __uint_as_float(v1[j]), square, sb, mf, inv, hi, 0.f);
              v0[j] = __float_as_uint(rj);
              v1[j] = square ? 0u : v0[j];
            }
            tmem_st16(lane_addr + c, v0);
            tmem_st16(lane_addr + kAccCols + c, v1);
          } else if (row < ctx.m) {
            const int64_t cc = col0 + c;
            int16_t* dst = rrow + cc * ctx.ldr;
            const int ncol = ctx.n - cc < 16 ? static_cast<int>(ctx.n - cc) : 16;
            if (SHORT1 && ncol == 16 && square) {  // k ≤ 128: one short slab, every modulus
#pragma unroll
              for (int j = 0; j < 16; ++j) {
                const float rj =
                    combine_residue_short1<true>(__uint_as_float(v0[j]), __uint_as_float(v1[j]), sb, mf, inv, hi);
                *dst = static_cast<int16_t>(as_i16_bits(rj));
                dst += ctx.ldr;
              }
            } else if (SHORT1 && ncol == 16) {
#pragma unroll
              for (int j = 0; j < 16; ++j) {
                const float rj =
                    combine_residue_short1<false>(__uint_as_float(v0[j]), __uint_as_float(v1[j]), sb, mf, inv, hi);
                *dst = static_cast<int16_t>(as_i16_bits(rj));
                dst += ctx.ldr;
              }
            } else if (!SHORT1 && ncol == 16 && short_slab) {  // a single short slab
#pragma unroll
              for (int j = 0; j < 16; ++j) {
                const float rj =
                    combine_residue_short(__uint_as_float(v0[j]), __uint_as_float(v1[j]), square, sb, mf, inv, hi);
                *dst = static_cast<int16_t>(as_i16_bits(rj));
                dst += ctx.ldr;
              }
            } else if (ncol == 16) {  // the common case: a full chunk
#pragma unroll
              for (int j = 0; j < 16; ++j) {
                const float rj =
                    combine_residue(__uint_as_float(v0[j]), __uint_as_float(v1[j]), square, sb, mf, inv, hi, 0.f);
                *dst = static_cast<int16_t>(as_i16_bits(rj));
                dst += ctx.ldr;
              }
            } else {
#pragma unroll
              for (int j = 0; j < 16; ++j) {
                const float rj =
                    combine_residue(__uint_as_float(v0[j]), __uint_as_float(v1[j]), square, sb, mf, inv, hi, 0.f);
                if (j < ncol) dst[j * ctx.ldr] = static_cast<int16_t>(as_i16_bits(rj));
              }
            }
          }
        }
        if (carry) {  // the written-back residues are in place before the next slab's MMAs
          tmem_st_wait();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_remote(acc_empty_leader);
        }
        accph ^= 1;
      }
      if (MODE == 1 && !SHORT1 && ok) {
        // rows past m hold zeros (TMA fills out-of-range rows with 0)
        if (row < ctx.m) atomicMax(reinterpret_cast<int*>(ctx.urow) + row, __float_as_int(rowmax));
        const int wm = __reduce_max_sync(0xffffffffu, __float_as_int(rowmax));
        if (lane == 0) atomicMax(&ctx.dev->u_max_bits, wm);
      }
    }
    if (!ok) {
      ctx.dev->status = kStatusTimeout;
      ctx.dev->timeout_site = 3;
    }
  }
  tc_fence_before();
  cluster_sync_all();  // neither CTA leaves while the pair's MMAs or loads may touch it
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem, kTmemCols);
}

// ---------------------------------------------------------------------------
// Tensor-pipe rate probe.  Every CTA pair issues `iters` MMAs of the residue
// GEMM's own form (cta_group::2, kind::f8f6f4, M = N = 256, K = 32) on one
// zero-filled operand tile pair in shared memory, into one accumulator, with
// no loads and no epilogue.  Timed by the caller, it gives the dense FP8 rate
// of the tensor pipes at the clock they run at: the ceiling for the residue
// GEMM, which issues the same instruction.  The shared-memory request keeps
// one CTA per SM, as in the GEMM.
// ---------------------------------------------------------------------------
constexpr int kProbeThreads = 64;
constexpr size_t kProbeSmem = 1024 + 2 * kTileBytes + 64 + 128 * 1024;

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kProbeThreads, 1)
    mma_rate_kernel(int64_t iters, Oz2Device* dev) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + 2 * kTileBytes);
  __shared__ uint32_t tmem_base_s;
  const int warp = threadIdx.x >> 5;
  const bool leader = cluster_ctarank() == 0;
  for (int i = threadIdx.x; i < 2 * kTileBytes / 16; i += kProbeThreads)
    reinterpret_cast<uint4*>(smem)[i] = make_uint4(0u, 0u, 0u, 0u);
  fence_proxy_async_smem();  // the tensor core reads what the threads wrote
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(bar), 1);
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(&tmem_base_s), kAccCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  if (leader && threadIdx.x == 32) {
    constexpr uint32_t idesc = idesc_f8_f32(kTileM, kTileN);
    const uint64_t a = smem_desc_sw128(smem_u32(smem)), b = a + (kTileBytes >> 4);
    for (int64_t it = 0; it < iters; ++it) {
      const uint32_t kk = static_cast<uint32_t>(it & 3);
      mma_f8_pair(tmem, a + 2 * kk, b + 2 * kk, idesc, it ? 1u : 0u);
    }
    mma_commit_pair(smem_u32(bar));
    if (!mbar_wait_bounded(smem_u32(bar), 0, kWaitLimit)) {
      dev->status = kStatusTimeout;
      dev->timeout_site = 4;
    }
  }
  __syncwarp();
  tc_fence_before();
  cluster_sync_all();  // the pair's MMAs read both CTAs' shared memory
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem, kAccCols);
}

cudaError_t launch_mma_rate(int64_t iters, Oz2Device* dev, int* pairs_out, cudaStream_t st);

// ---------------------------------------------------------------------------
// Plain CUDA-core kernel with the same semantics (diagnostic reference for
// the tensor-core path; accumulates the same integer plane products in FP32
// in sequential k order, so exactness follows from the same bound).
// ---------------------------------------------------------------------------
template <int MODE>
__global__ void plane_gemm_simt_kernel(const uint8_t* __restrict__ pa, const uint8_t* __restrict__ pb,
                                       const __grid_constant__ Oz2Moduli mods, int64_t k_pad, EpiCtx ctx) {
  const int64_t row = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const int64_t col = blockIdx.y;
  if (row >= ctx.m || col >= ctx.n) return;
  const uint8_t* ar = pa + row * k_pad;
  const uint8_t* bc = pb + col * k_pad;
  if (MODE == 1) {  // magnitude planes: one plane, rows × k_pad
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
    const float hi = static_cast<float>(mods.m[i] - 1 - mods.m[i] / 2);
    const int64_t slab = square ? kKSlabSquare : kKSlabMerged;
    // Byte l of plane plane_off + j of row `rw` (of A) or column (of B), in
    // 128 × 128-byte blocks.
    const int64_t kblocks = k_pad / kPlaneLine;
    auto plane = [&](const uint8_t* base, int64_t rw, int j, int64_t l) {
      const int64_t blk = ((rw / kPlaneRows) * kblocks + l / kPlaneLine) * mods.nplanes + mods.plane_off[i] + j;
      return e4m3_to_float(base[blk * kPlaneBlock + (rw % kPlaneRows) * kPlaneLine + l % kPlaneLine]);
    };
    float res = 0.f;
    for (int64_t l0 = 0; l0 < k_pad; l0 += slab) {
      float a0 = 0.f, a1 = 0.f;
      const int64_t l1 = min(k_pad, l0 + slab);
      for (int64_t l = l0; l < l1; ++l) {
        const float x0 = plane(pa, row, 0, l), y0 = plane(pb, col, 0, l);
        const float x1 = plane(pa, row, 1, l), y1 = plane(pb, col, 1, l);
        if (square) {
          a0 += x0 * y0;
          a1 += x1 * y0 + x0 * y1;
        } else {
          const float x2 = plane(pa, row, 2, l), y2 = plane(pb, col, 2, l);
          a0 += x0 * y0;
          a1 += x1 * y1 + x2 * y2;
        }
      }
      res = combine_residue(a0, a1, square, static_cast<float>(mods.sq_base[i]), mf, inv, hi, res);
    }
    ctx.res[static_cast<size_t>(i) * ctx.n * ctx.ldr + col * ctx.ldr + row] = static_cast<int16_t>(res);
  }
}

// ---------------------------------------------------------------------------
// Host side: tensor maps and launch.
// ---------------------------------------------------------------------------
// Magnitude plane of one operand: rows × k_pad bytes, row-major; the box is
// 128 rows × 128 bytes with the 128-byte swizzle the MMA descriptors use.
static bool make_plane_map(CUtensorMap* map, const uint8_t* base, int64_t rows, int64_t k_pad) {
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(k_pad), static_cast<cuuint64_t>(rows), 1};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(k_pad), static_cast<cuuint64_t>(rows * k_pad)};
  cuuint32_t box[3] = {kBK, static_cast<cuuint32_t>(kRows), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<uint8_t*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// ---------------------------------------------------------------------------
// Split K.  A problem whose units fill few waves of the CTA pairs (a small C
// with a long k) runs each unit's k-blocks in kparts parts; the parts'
// residues land in scratch planes [part][modulus][column][row] and
// fold_parts_kernel sums them mod m into C^(i).
// ---------------------------------------------------------------------------
constexpr int kFoldThreads = 128;

// C^(i) from its parts: the sum of kparts centred residues has magnitude at
// most kparts·⌊m/2⌋ < 2^16, so centred_small reduces it exactly.  One thread
// takes 8 consecutive rows of one column (16-byte loads: ldr is a multiple
// of 8 and both buffers are 16-byte aligned); blockIdx.z is the modulus.
__global__ void __launch_bounds__(kFoldThreads) fold_parts_kernel(const int16_t* __restrict__ part,
                                                                  int16_t* __restrict__ res, int64_t m, int64_t n,
                                                                  int64_t ldr, int kparts,
                                                                  const __grid_constant__ Oz2Moduli mods) {
  const int i = blockIdx.z;
  const float mf = static_cast<float>(mods.m[i]), inv = 1.f / mf;
  const float hi = static_cast<float>(mods.m[i] - 1 - mods.m[i] / 2);
  const int64_t row0 = (static_cast<int64_t>(blockIdx.x) * kFoldThreads + threadIdx.x) * 8;
  if (row0 >= m) return;
  const size_t plane = static_cast<size_t>(n) * ldr, pstride = static_cast<size_t>(mods.r) * plane;
  for (int64_t col = blockIdx.y; col < n; col += gridDim.y) {
    const size_t off = static_cast<size_t>(i) * plane + static_cast<size_t>(col) * ldr + row0;
    if (row0 + 8 <= m) {
      int acc[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[j] = 0;
      for (int p = 0; p < kparts; ++p) {
        const uint4 v = __ldg(reinterpret_cast<const uint4*>(part + p * pstride + off));
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          acc[2 * j] += static_cast<int16_t>(w[j] & 0xFFFFu);
          acc[2 * j + 1] += static_cast<int>(w[j]) >> 16;
        }
      }
      uint32_t o[4];
#pragma unroll
      for (int j = 0; j < 4; ++j)
        o[j] = as_i16_bits(centred_small(static_cast<float>(acc[2 * j]), mf, inv, hi)) |
               (as_i16_bits(centred_small(static_cast<float>(acc[2 * j + 1]), mf, inv, hi)) << 16);
      *reinterpret_cast<uint4*>(res + off) = make_uint4(o[0], o[1], o[2], o[3]);
    } else {
      for (int64_t r = row0; r < m; ++r) {
        int a = 0;
        for (int p = 0; p < kparts; ++p) a += part[p * pstride + off + (r - row0)];
        res[off + (r - row0)] = static_cast<int16_t>(as_i16_bits(centred_small(static_cast<float>(a), mf, inv, hi)));
      }
    }
  }
}

// At most 16 parts of k.  The fold's sum of kparts centred residues stays
// far inside 16 bits (16·⌊m/2⌋ ≤ 8704); what limits a split in practice is
// the scratch (the magnitude-plane region must hold kparts partial residue
// sets) and the cost model's 5% gain rule.
constexpr int64_t kMaxKParts = 16;
constexpr int64_t kMinPartSteps = 4;   // k-blocks (512 k-entries) per part at least

// Estimated duration of the residue GEMM under the unit schedule (nonsquare
// moduli first, waves dealt in alternating directions), in units of one
// stage pair on a CTA pair (a 256×256×128 FP8 product, about 0.39 µs at
// 2.07 GHz): the largest load over the pairs.  A nonsquare unit of s
// k-blocks costs 3s plus 10 per epilogue drain (one per 4096 k-entries), a
// square one 2s plus 10 per 32768.  A split adds the fold (its bytes at
// about 5 TB/s, and a launch).  The pairs' loads are piecewise constant in
// the pair index, changing only where the heavy units and all units end in
// their last waves, so those pairs and the two ends cover the maximum.
static double split_cost(int64_t ntiles, int r, int nsq, int64_t ksteps, int64_t kparts, int64_t pairs, int64_t m,
                         int64_t n) {
  const int64_t s = (ksteps + kparts - 1) / kparts;
  const int64_t U = ntiles * r * kparts, H = ntiles * (r - nsq) * kparts;
  const int64_t P = std::max<int64_t>(1, std::min(pairs, U));
  constexpr int64_t kSlabM = kKSlabMerged / kBK, kSlabS = kKSlabSquare / kBK;
  const double wh = 3.0 * s + 10.0 * ((s + kSlabM - 1) / kSlabM);
  const double wl = 2.0 * s + 10.0 * ((s + kSlabS - 1) / kSlabS);
  auto count = [&](int64_t X, int64_t q) {  // units below X that pair q takes
    const int64_t w0 = X / P, rem = X - w0 * P;
    const int64_t pos = (w0 & 1) ? P - 1 - q : q;
    return w0 + (pos < rem ? 1 : 0);
  };
  auto load = [&](int64_t q) {
    const int64_t h = count(H, q);
    return h * wh + (count(U, q) - h) * wl;
  };
  double mx = std::max(load(0), load(P - 1));
  for (const int64_t X : {H, U}) {
    const int64_t w0 = X / P, rem = X - w0 * P;
    const int64_t b = (w0 & 1) ? P - rem : rem;
    for (const int64_t q : {b - 1, b})
      if (q >= 0 && q < P) mx = std::max(mx, load(q));
  }
  if (kparts > 1) mx += (3.0 + (kparts + 1.0) * r * m * n * 2.0 / 5.0e6) / 0.39;
  return mx;
}

// Parts of K per residue-GEMM unit: 1 unless the units fill fewer than four
// waves and a split of at most max_parts (each part non-empty and at least
// kMinPartSteps k-blocks) is estimated at least 5% faster.
static int64_t choose_kparts(int64_t ntiles, int r, int nsq, int64_t ksteps, int64_t pairs, int64_t m, int64_t n,
                             int64_t max_parts) {
  if (max_parts < 2 || ntiles * r >= 4 * pairs) return 1;
  int64_t best = 1;
  double best_cost = split_cost(ntiles, r, nsq, ksteps, 1, pairs, m, n);
  for (int64_t p = 2; p <= max_parts; ++p) {
    const int64_t s = (ksteps + p - 1) / p;
    if (s < kMinPartSteps) break;
    if ((ksteps + s - 1) / s != p) continue;  // a part would be empty
    const double c = split_cost(ntiles, r, nsq, ksteps, p, pairs, m, n);
    if (c < 0.95 * best_cost) {
      best = p;
      best_cost = c;
    }
  }
  return best;
}

int64_t residue_gemm_kparts(int64_t m, int64_t n, int64_t k_pad, int r, int nsq, int64_t ldr, size_t partial_bytes,
                            int64_t pairs) {
  if (m <= 0 || n <= 0 || k_pad <= 0 || r < 1 || ldr < m || ldr % 8 != 0 || pairs < 1) return 1;
  const size_t part_bytes = static_cast<size_t>(r) * n * ldr * sizeof(int16_t);
  const int64_t max_parts = std::min<int64_t>(kMaxKParts, static_cast<int64_t>(partial_bytes / part_bytes));
  const int64_t ntiles = ((m + kTileM - 1) / kTileM) * ((n + kTileN - 1) / kTileN);
  return choose_kparts(ntiles, r, nsq, k_pad / kBK, pairs, m, n, max_parts);
}

static size_t gemm_smem_bytes() { return 1024 + static_cast<size_t>(kStages) * kStageBytes + 8 * (2 * kStages + 3); }

// The magnitude GEMM split along k: each part adds its tiles' partial sums
// into U with 16-byte vector atomics (every partial sum is an integer number
// of units 2^-2c below 2^24, like the whole sum, so FP32 adds them exactly in
// any order), and this kernel then takes each row's maximum, as the unsplit
// epilogue does: a warp per row of the row-major U.
constexpr int kRowMaxThreads = 256;
__global__ void __launch_bounds__(kRowMaxThreads) plus_one_rowmax_kernel(const float* __restrict__ U, int64_t m,
                                                                         int64_t n, int64_t ldu,
                                                                         float* __restrict__ urow, Oz2Device* dev) {
  const int lane = threadIdx.x & 31;
  const int64_t row = static_cast<int64_t>(blockIdx.x) * (kRowMaxThreads / 32) + (threadIdx.x >> 5);
  if (row >= m) return;  // whole warps
  float mx = 0.f;
  const float* p = U + row * ldu;
  for (int64_t col = lane; col < n; col += 32) mx = fmaxf(mx, __ldg(p + col));
  const int wm = __reduce_max_sync(0xffffffffu, __float_as_int(mx));  // nonnegative floats order as their bits
  if (lane == 0) {
    atomicMax(reinterpret_cast<int*>(urow) + row, wm);
    atomicMax(&dev->u_max_bits, wm);
  }
}

// Parts of k for the magnitude GEMM: its 256×256 tiles fill fewer than half
// a wave of the CTA pairs only for a small C with a long k; then each tile
// runs in as many parts as the pairs allow (at most 64, each at least
// kMinPartSteps k-blocks), and U's partial sums go through scratch.
static int64_t magnitude_ldu(int64_t n) { return (n + 3) / 4 * 4; }

static int64_t magnitude_kparts(int64_t ntiles, int64_t ksteps, int64_t pairs, int64_t m, int64_t n,
                                size_t scratch_bytes) {
  if (2 * ntiles >= pairs || scratch_bytes < static_cast<size_t>(m) * magnitude_ldu(n) * sizeof(float)) return 1;
  int64_t p = std::min<int64_t>({64, pairs / ntiles, ksteps / kMinPartSteps});
  if (p < 2) return 1;
  const int64_t s = (ksteps + p - 1) / p;
  return (ksteps + s - 1) / s;  // no empty part
}

int64_t magnitude_gemm_kparts(int64_t m, int64_t n, int64_t k_pad, size_t scratch_bytes, int64_t pairs) {
  if (m <= 0 || n <= 0 || k_pad <= 0 || pairs < 1) return 1;
  const int64_t ntiles = ((m + kTileM - 1) / kTileM) * ((n + kTileN - 1) / kTileN);
  return magnitude_kparts(ntiles, k_pad / kBK, pairs, m, n, scratch_bytes);
}

// mode: 0 residues (tensor cores), 1 magnitude (tensor cores),
//       2 residues (SIMT reference), 3 magnitude (SIMT reference).
cudaError_t launch_plane_gemm(int64_t m, int64_t n, int64_t k_pad, const Oz2Moduli& mods,
                              const uint8_t* planes_a, const uint8_t* planes_b, int mode,
                              int16_t* residues, int64_t ldr, float* urow, Oz2Device* dev, cudaStream_t st,
                              int16_t* partials, size_t partial_bytes) {
  if (m == 0 || n == 0) return cudaSuccess;
  EpiCtx ctx{residues, urow, dev, m, n, ldr, nullptr, 0};
  if (mode >= 2) {
    dim3 g(static_cast<unsigned>((m + 127) / 128), static_cast<unsigned>(n));
    count_launch();
    if (mode == 2) plane_gemm_simt_kernel<0><<<g, 128, 0, st>>>(planes_a, planes_b, mods, k_pad, ctx);
    else plane_gemm_simt_kernel<1><<<g, 128, 0, st>>>(planes_a, planes_b, mods, k_pad, ctx);
    return cudaGetLastError();
  }
  CUtensorMap ta, tb;
  const bool maps = mode == 0 ? make_block_map(&ta, planes_a, m, k_pad, mods.nplanes) &&
                                    make_block_map(&tb, planes_b, n, k_pad, mods.nplanes)
                              : make_plane_map(&ta, planes_a, m, k_pad) && make_plane_map(&tb, planes_b, n, k_pad);
  if (!maps) return cudaErrorInvalidValue;
  UnitMap um;
  um.ntm = (m + kTileM - 1) / kTileM;
  um.ntn = (n + kTileN - 1) / kTileN;
  um.ntiles = um.ntm * um.ntn;
  um.nunits = um.ntiles * (mode == 0 ? mods.r : 1);
  // Square moduli lead the set; the nonsquare ones are scheduled first.
  um.nsq = 0;
  while (um.nsq < mods.r && mods.sq_base[um.nsq]) ++um.nsq;
  um.nheavy = mode == 0 ? mods.r - um.nsq : 0;
  for (int i = um.nsq; i < mods.r; ++i)
    if (mods.sq_base[i]) um.nheavy = 0;  // not a prefix: keep the index order
  um.ksteps = k_pad / kBK;
  um.kparts = 1;
  um.kpart_steps = um.ksteps;
  const size_t smem = gemm_smem_bytes();
  auto kern = mode == 1 ? plane_gemm_kernel<1> : k_pad == kBK ? plane_gemm_kernel<0, true> : plane_gemm_kernel<0>;
  cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (err != cudaSuccess) return err;
  // Persistent grid: as many CTA pairs as can be resident at once.
  int64_t pairs = num_sms() / 2;
  {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(2 * pairs));
    cfg.blockDim = dim3(kGemmThreads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = 2;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    int clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&clusters, kern, &cfg) == cudaSuccess && clusters > 0)
      pairs = std::min<int64_t>(pairs, clusters);
    else
      cudaGetLastError();
  }
  // Split K where the scratch holds the parts (16-byte aligned rows: the
  // fold reads and writes 8 residues at a time).
  if (mode == 0 && partials && reinterpret_cast<uintptr_t>(partials) % 16 == 0 &&
      reinterpret_cast<uintptr_t>(residues) % 16 == 0) {
    const int nheavy_sq = um.nheavy ? um.nsq : mods.r;  // the model's squares
    um.kparts = residue_gemm_kparts(m, n, k_pad, mods.r, nheavy_sq, ldr, partial_bytes, pairs);
    um.kpart_steps = (um.ksteps + um.kparts - 1) / um.kparts;
    um.nunits *= um.kparts;
    if (um.kparts > 1) ctx.res = partials;
  }
  // The magnitude GEMM of a small C with a long k: parts of k, with U's
  // partial sums in the scratch (`partials`, 16-byte aligned).
  if (mode == 1 && partials && reinterpret_cast<uintptr_t>(partials) % 16 == 0) {
    um.kparts = magnitude_kparts(um.ntiles, um.ksteps, pairs, m, n, partial_bytes);
    um.kpart_steps = (um.ksteps + um.kparts - 1) / um.kparts;
    um.nunits *= um.kparts;
    if (um.kparts > 1) {
      kern = plane_gemm_kernel<1, true>;  // same shared memory and threads, so the same pairs fit
      err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
      if (err != cudaSuccess) return err;
      ctx.upart = reinterpret_cast<float*>(partials);
      ctx.ldu = magnitude_ldu(n);
      err = cudaMemsetAsync(ctx.upart, 0, static_cast<size_t>(m) * ctx.ldu * sizeof(float), st);
      if (err != cudaSuccess) return err;
    }
  }
  pairs = std::max<int64_t>(1, std::min<int64_t>(pairs, um.nunits));
  count_launch();
  kern<<<static_cast<unsigned>(2 * pairs), kGemmThreads, smem, st>>>(ta, tb, mods, k_pad, um, ctx);
  if (ctx.upart) {
    count_launch();
    constexpr int64_t rows_per_block = kRowMaxThreads / 32;
    plus_one_rowmax_kernel<<<static_cast<unsigned>((m + rows_per_block - 1) / rows_per_block), kRowMaxThreads, 0,
                             st>>>(ctx.upart, m, n, ctx.ldu, urow, dev);
  }
  if (mode == 0 && um.kparts > 1) {  // the residue GEMM's parts, folded into C^(i)
    const int64_t row_threads = (m + 7) / 8;
    dim3 g(static_cast<unsigned>((row_threads + kFoldThreads - 1) / kFoldThreads),
           static_cast<unsigned>(std::min<int64_t>(n, 32768)), static_cast<unsigned>(mods.r));
    count_launch();
    fold_parts_kernel<<<g, kFoldThreads, 0, st>>>(partials, residues, m, n, ldr, static_cast<int>(um.kparts), mods);
  }
  return cudaGetLastError();
}

// The rate probe on as many CTA pairs as can be resident at once.
cudaError_t launch_mma_rate(int64_t iters, Oz2Device* dev, int* pairs_out, cudaStream_t st) {
  cudaError_t err =
      cudaFuncSetAttribute(mma_rate_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kProbeSmem));
  if (err != cudaSuccess) return err;
  int64_t pairs = num_sms() / 2;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(2 * pairs));
  cfg.blockDim = dim3(kProbeThreads);
  cfg.dynamicSmemBytes = kProbeSmem;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = 2;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  int clusters = 0;
  if (cudaOccupancyMaxActiveClusters(&clusters, mma_rate_kernel, &cfg) == cudaSuccess && clusters > 0)
    pairs = std::min<int64_t>(pairs, clusters);
  else
    cudaGetLastError();
  if (pairs_out) *pairs_out = static_cast<int>(pairs);
  count_launch();
  mma_rate_kernel<<<static_cast<unsigned>(2 * pairs), kProbeThreads, kProbeSmem, st>>>(iters, dev);
  return cudaGetLastError();
}

}  // namespace oz2
