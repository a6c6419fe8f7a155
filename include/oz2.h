/*
 * oz2.h -- C ABI of liboz2: FP64 matrix multiplication emulated with Ozaki
 * Scheme II on FP8 (E4M3) tensor cores, for one NVIDIA GB300 (sm_103a).
 *
 * The method (arxiv 2606.06510, §2.3-2.5, Algorithm 1):
 *   1. choose power-of-two row/column scales D, E and form the integer
 *      matrices Ã = ⌊DA⌉, B̃ = ⌊BE⌉                          (Eq. scale)
 *   2. for r pairwise-coprime moduli m_i, store the centred residues of Ã
 *      and B̃ as E4M3 digit planes and form C^(i) = Ã B̃ mod m_i with three
 *      FP8 plane products per modulus                 (Eq. modgemm, §2.5)
 *   3. rebuild C̃ = ÃB̃ with Garner's algorithm and return D^-1 C̃ E^-1
 *                                                      (Eq. garner, App. A)
 * Rows of A (columns of B) holding a non-finite value, or whose exponent is
 * far from the others, take a native FP64 path (Algorithm 1, fallback).
 *
 * Conventions shared by every entry point:
 *  - Matrices are column-major, as in BLAS.  A is m×k (leading dimension
 *    lda ≥ max(1,m)), B is k×n (ldb ≥ max(1,k)), C is m×n (ldc ≥ max(1,m)).
 *  - Pointers named d_* are device pointers; h_* are host pointers.  The
 *    caller owns every buffer it passes; the library never frees them.
 *  - `stream` is a cudaStream_t (NULL = the legacy default stream).  Work is
 *    enqueued asynchronously; no entry point synchronises the host on the
 *    success path unless its comment says so.
 *  - Return value: OZ2_OK or a negative oz2_status.  Errors detected on the
 *    host are returned immediately and nothing is enqueued.  Errors raised by
 *    a kernel (a bounded wait that timed out) are recorded in a device status
 *    word read by oz2_get_stats()/oz2_check_device_status().
 *  - num_moduli r ∈ [1, 16]: the first r moduli of the paper's set S
 *    (1089, 1024, 961, 841, 625, 529, 511, 509, 503, 499, 491, 487; §2.5),
 *    extended for r > 12 by 479, 467, 463, 461.  r = 12 is the paper's
 *    working point; r = 13 is needed for FP64-level accuracy at large k.
 */
#ifndef OZ2_H
#define OZ2_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  OZ2_OK = 0,
  OZ2_ERR_INVALID_ARG = -1,   /* a size, leading dimension or pointer is invalid */
  OZ2_ERR_UNSUPPORTED_R = -2, /* num_moduli outside [1, 16] */
  OZ2_ERR_ALLOC = -3,         /* workspace allocation failed or too small */
  OZ2_ERR_CUDA = -4,          /* a CUDA runtime call or launch failed */
  OZ2_ERR_TIMEOUT = -5,       /* a device-side bounded wait expired */
  OZ2_ERR_UNSUPPORTED = -6    /* a size beyond the implemented limits */
} oz2_status;

/* Quantiser of Eq. (scale), Table "numerical-contract variants". */
typedef enum { OZ2_QUANT_TZ = 0, OZ2_QUANT_RN = 1 } oz2_quant;

/* Scale choice.  R2 (default): per-row/column power-of-two scales from the
 * "+1" max-magnitude GEMM U = ÂB̂ (§2.4), so that Σ_l|Ã_il||B̃_lj| ≤ 2^T < M/2.
 * R1: the crude bound μ = k·max|Ã|·max|B̃| of Algorithm 1 (no "+1" GEMM). */
typedef enum { OZ2_SCALE_R2 = 0, OZ2_SCALE_R1 = 1 } oz2_scale_mode;

/* Flags for oz2_dgemm_ex. */
#define OZ2_FLAG_NO_FALLBACK 0x1u   /* flag only non-finite rows/columns */
#define OZ2_FLAG_TIMING      0x2u   /* record per-stage CUDA events on the stream;
                                       harvested by oz2_get_stats (no host sync
                                       inside the call) */
/* For num_moduli 11 or 12 and k ≤ 256: run the residue GEMM and the
 * reconstruction fused in one kernel, each output's residues folded into
 * its CRT sum on chip (Algorithm 1 Phase 3 in the GEMM epilogue), instead of
 * two launches through the residue matrices.  It moves fewer DRAM bytes
 * (no 2r bytes per output written and read back) but streams every plane of
 * A through L2 once per 32 columns of C, and on one GB300 it measured slower
 * than the two launches for every shape tried; see oz2_dgemm_ex. */
#define OZ2_FLAG_FUSED       0x4u
/* For a skinny C (n ≤ 32, m ≥ 128, k padded to 1024 or more): form A's
 * digit planes on chip from A inside the residue GEMM (plane storage mode F,
 * §"plane-storage modes"), so they are never written to device memory and
 * read back, instead of storing them.  It moves fewer DRAM bytes but runs
 * the conversion on one CTA per 128 rows of A; on one GB300 the batched
 * GEMV 16384 × 16 × 16384 took 5.12 ms this way against 4.55 ms with the
 * planes stored, so it is not the default.  Ignored where it does not
 * apply; see oz2_dgemm_ex. */
#define OZ2_FLAG_ON_THE_FLY  0x8u
/* Diagnostic only: run the "+1" and residue plane GEMMs on CUDA cores with
 * the same integer plane products and epilogue arithmetic (slow; used by
 * the tests to separate tensor-core issues from the rest of the path). */
#define OZ2_FLAG_DEBUG_SIMT_GEMM 0x100u

/* Statistics of the most recent oz2_dgemm / oz2_dgemm_ex call on this
 * device.  Reading them synchronises the device. */
typedef struct {
  int32_t status;            /* device status word: 0, or an oz2_status */
  int32_t fallback_rows;     /* rows of A that took the native FP64 path */
  int32_t fallback_cols;     /* columns of B that took the native FP64 path */
  int32_t u_max;             /* max_i u_i of the "+1" pass (R2) */
  int32_t s;                 /* common column budget s (R2), or pB (R1) */
  int32_t d_min, d_max;      /* range of the row exponents d_i */
  int32_t e_min, e_max;      /* range of the column exponents e_j */
  int32_t k_slab;            /* K-slab of exact FP32 accumulation used */
  float stage_ms[8];         /* mean per call of: scan, magnitude planes,
                                "+1" GEMM, scale choice, deconstruct, residue
                                GEMM, CRT, fallback -- over the calls made
                                with OZ2_FLAG_TIMING since the last read */
  int32_t timed_calls;       /* number of calls averaged in stage_ms */
  int64_t kernel_launches;   /* kernels launched by the library since the
                                last read (all devices) */
} oz2_stats;

/* ---------------------------------------------------------------------
 * Production entry points
 * ------------------------------------------------------------------- */

/* C = A·B (overwrite, β = 0) by Ozaki Scheme II with TZ quantiser and R2
 * scales.  Allocates its workspace stream-ordered on `stream` from the
 * library's memory pool (see oz2_trim_memory) and frees it on the same
 * stream.  m == 0 or n == 0: no-op; k == 0: C = 0. */
int oz2_dgemm(int64_t m, int64_t n, int64_t k,
              const double* d_A, int64_t lda,
              const double* d_B, int64_t ldb,
              double* d_C, int64_t ldc,
              int num_moduli, void* stream);

/* As oz2_dgemm with A, B and C in HOST memory (pinned memory gives the
 * best transfer rate).  Copies A and B to the device, computes, copies C
 * back, and synchronises `stream` before returning.  Device buffers and the
 * workspace are allocated and freed stream-ordered inside the call, from the
 * library's memory pool.  A contiguous matrix (ld = rows) moves in one
 * linear copy, any other in a pitched copy.  The copies run on a
 * library-owned copy stream: B first, then A in up to 4 column chunks (of
 * at least 32 MB); B's scan, flags and magnitude planes run while A is
 * copied, and A's scan chunk by chunk as its columns arrive.  The residue
 * GEMM, reconstruction and fallback then run by column blocks (oz2_plan's
 * host_widths), and each block of C is copied back on the copy stream while
 * the next block is computed.  The result is the same as one oz2_dgemm on
 * device copies.  Host-buffer calls on one device share the copy stream and
 * are serialised. */
int oz2_dgemm_host(int64_t m, int64_t n, int64_t k,
                   const double* h_A, int64_t lda,
                   const double* h_B, int64_t ldb,
                   double* h_C, int64_t ldc,
                   int num_moduli, void* stream);

/* As oz2_dgemm, for callers that must not allocate device memory (a host
 * framework whose allocator owns all device memory, code that may not block
 * or fail on an allocation at run time, plug-ins handed only their input and
 * output buffers).  The paper has no counterpart: this is a deployment
 * variant of the same computation.  Instead of allocating a workspace it uses
 * a fixed 32 MiB array in the library's own device memory (held on every GPU
 * that loads the library until the process exits); problems whose
 * oz2_workspace_size exceeds 32 MiB (about 512³ at num_moduli = 16) return
 * OZ2_ERR_UNSUPPORTED.  It calls no allocation routine and creates no memory
 * pool (the library's stream-ordered pool is made only by the entry points
 * that allocate).  The first call on each device looks up the array's device
 * address and uploads the library's digit-plane table with synchronous
 * copies; make that first call before any stream capture.  All
 * calls share the one array: calls whose work overlaps on the GPU (different
 * streams, or concurrent host threads) race and must be serialised by the
 * caller.  Each call clears what it needs before using it. */
int oz2_dgemm_noalloc(int64_t m, int64_t n, int64_t k,
                      const double* d_A, int64_t lda,
                      const double* d_B, int64_t ldb,
                      double* d_C, int64_t ldc,
                      int num_moduli, void* stream);

/* Bytes of device workspace oz2_dgemm_ex needs for this problem. */
size_t oz2_workspace_size(int64_t m, int64_t n, int64_t k, int num_moduli);

/* As oz2_dgemm, with an explicit quantiser (oz2_quant), scale mode
 * (oz2_scale_mode), flags (OZ2_FLAG_*) and caller-provided device workspace of
 * ws_bytes ≥ oz2_workspace_size(...) bytes, 256-byte aligned.  After the
 * call the workspace holds the intermediates at the offsets reported by
 * oz2_workspace_layout (they stay valid until the workspace is reused).
 * With OZ2_FLAG_FUSED, num_moduli 11 or 12 and k ≤ 256 (k padded to 256 or
 * less) the residue GEMM and the reconstruction run fused; the residues
 * region then holds that kernel's scratch instead of the residue matrices.
 * With OZ2_FLAG_ON_THE_FLY and a skinny C (n ≤ 32, m ≥ 128, k padded to
 * 1024 or more) A's digit planes are formed on chip from A inside the
 * residue GEMM and never stored (the planes_a region is then left
 * unwritten).  The result C is the same on every path, bit for bit. */
int oz2_dgemm_ex(int64_t m, int64_t n, int64_t k,
                 const double* d_A, int64_t lda,
                 const double* d_B, int64_t ldb,
                 double* d_C, int64_t ldc,
                 int num_moduli, int quant, int scale, unsigned flags,
                 void* d_workspace, size_t ws_bytes, void* stream);

/* Byte offsets of the intermediates inside the oz2_dgemm_ex workspace.
 * Layouts (all written by the library):
 *   ra[m], cb[n]          int32  row/column max-exponents (|x| < 2^e)
 *   row_flag[m], col_flag[n] uint8  bit0 fallback, bit1 zero in emulation
 *   d[m], e[n]            int32  the scale exponents (D = diag 2^d_i ...)
 *   urow[m]               float  max_j U_ij of the "+1" GEMM (R2)
 *   mag_a, mag_b          uint8  magnitude planes Â (m×k_pad), B̂ (n×k_pad),
 *                                row-major.  When the residue GEMM splits K
 *                                (a small C with a long k) this region is
 *                                then reused for the partial residues, so
 *                                after such a call it holds those instead.
 *   planes_a, planes_b    uint8  E4M3 digit planes, see oz2_plane_layout
 *   residues              int16  r matrices C^(i), each m×n column-major
 *                                with ld = res_ld (matrix i starts at element
 *                                i·n·res_ld), centred in
 *                                [-⌊m_i/2⌋, m_i-1-⌊m_i/2⌋]; after a fused
 *                                call (see oz2_dgemm_ex) the fused kernel's
 *                                scratch instead
 */
typedef struct {
  size_t ra, cb, row_flag, col_flag, d, e, urow, misc;
  size_t mag_a, mag_b, planes_a, planes_b, residues, total;
  int64_t k_pad;             /* k rounded up to a multiple of 128 */
  int32_t num_planes;        /* stored planes per operand element */
  int64_t res_ld;            /* m rounded up to a multiple of 8 */
} oz2_ws_layout;
int oz2_workspace_layout(int64_t m, int64_t n, int64_t k, int num_moduli,
                         oz2_ws_layout* out);

/* How the library runs a problem on a GPU with cta_pairs CTA pairs (half its
 * SM count: 76 on a GB300).  Host arithmetic only: it touches no device and
 * runs without one.  A call on a device uses min(SMs/2, the residue GEMM's
 * resident two-CTA clusters) pairs, which is SMs/2 unless another kernel's
 * resources or a partitioned device cut the resident clusters; the plan
 * matches a call only for the pair count that call used.
 *   kparts        parts of k per residue-GEMM unit in oz2_dgemm_ex and
 *                 oz2_dgemm (1: no split).  A small C with a long k fills
 *                 few waves of the CTA pairs; each unit then covers 1/kparts
 *                 of the k-blocks, and a fold sums the parts' residues mod m.
 *   host_blocks   column blocks of oz2_dgemm_host (1 to 8).  The blocks run
 *                 the residue GEMM, reconstruction and fallback one after
 *                 another, each copied back while the next computes.
 *   host_widths   their widths: multiples of 256 but the last.  They
 *                 minimise the end of the last copy back on a model of the
 *                 call: each block's GEMM waves and reconstruction at this
 *                 library's rates on a GB300, its copy at 190 GB/s over the
 *                 host link, one copy at a time.  Long k gives a narrow last
 *                 block (its copy is the one left exposed); short k, where
 *                 the copies dominate, a narrow first one (the copies start
 *                 early).  Identical shapes reuse the last plan.
 *   host_kparts   the residue GEMM's kparts for each block.
 *   mag_kparts    parts of k of the "+1" magnitude GEMM (1: no split).
 *                 When its 256×256 tiles fill less than half a wave (a
 *                 small C with a long k), each tile runs in up to 64 parts
 *                 of at least 512 k-entries; the parts add their FP32 sums
 *                 (exact: integers in units of 2^-2c below 2^24) into an
 *                 m×n buffer in the then unused digit-plane region, and a
 *                 row-maximum kernel follows (one launch more).
 * Returns OZ2_OK, OZ2_ERR_INVALID_ARG (null out, negative sizes,
 * cta_pairs < 1) or OZ2_ERR_UNSUPPORTED_R. */
typedef struct {
  int64_t kparts;
  int32_t host_blocks;
  int64_t host_widths[8];
  int64_t host_kparts[8];
  int64_t mag_kparts;
} oz2_plan_info;
int oz2_plan(int64_t m, int64_t n, int64_t k, int num_moduli, int cta_pairs, oz2_plan_info* out);

/* Digit-plane layout (§2.5).  For operand X with `rows` rows (m for A, n
 * for B) there are P planes (the return value), each logically a rows×k_pad
 * byte matrix zero-padded from k to k_pad, stored as 128 × 128-byte blocks
 * with the rows padded to rows_pad = ⌈rows/128⌉·128 (pad rows hold zero
 * digits): byte l of row `row` of plane p is at
 *   ((⌊row/128⌋·(k_pad/128) + ⌊l/128⌋)·P + p)·16384 + (row mod 128)·128
 *     + (l mod 128),
 * so a plane buffer holds P·rows_pad·k_pad bytes, each block is one MMA
 * operand tile, and the P blocks of one (row block, k-block) are
 * consecutive.  The planes of modulus i are consecutive, starting at
 * plane_offset[i]:
 *   square m_i = s²:  (d0, d1)              d = d0 + s·d1, balanced base s
 *   nonsquare, B:     (d0+d1, d0, d1)       d = d0 + 16·d1, carry-corrected
 *   nonsquare, A:     (d0+d1, d0, -16·d1)   (pre-scaled for the merged
 *                                           accumulator d0e0 - 16·d1e1, §2.5)
 * where d is the centred residue of the integer Ã (or B̃) entry.  Each byte
 * is the E4M3 code of the integer digit.  Writes num_moduli offsets and
 * returns the total plane count. */
int oz2_plane_layout(int num_moduli, int32_t* plane_offset);

/* Statistics of the last call on the current device (synchronises; resets
 * the timing accumulators and the launch counter). */
int oz2_get_stats(oz2_stats* out);

/* Self-test of the failure path.  Launches one warp that waits on an
 * mbarrier nothing arrives at, bounded by limit_cycles SM cycles (1000 to
 * 4e9), and on expiry records OZ2_ERR_TIMEOUT in the device status word, as
 * every library kernel does when one of its waits expires.  The wait ends by
 * its bound: nothing faults or hangs.  The next oz2_check_device_status then
 * returns OZ2_ERR_TIMEOUT and clears the word.  OZ2_ERR_INVALID_ARG for a
 * limit out of range. */
int oz2_selftest_timeout(long long limit_cycles, void* stream);

/* Measurement probe for the FP8 tensor-pipe peak (the dense FP8 rate of the
 * paper's hardware table, here measured rather than quoted).  Every CTA pair
 * that can be resident issues `iters` (1 to 2^40) MMAs of the residue GEMM's
 * own form, tcgen05.mma.cta_group::2.kind::f8f6f4 with M = N = 256, K = 32,
 * on zero-filled operands in shared memory into one TMEM accumulator: no
 * loads, no epilogue, no output.  The caller times the launch on `stream`;
 * the work is (*cta_pairs)·iters·2·256·256·32 FP8 flops.  Writes the number
 * of CTA pairs to *cta_pairs (if not null).  OZ2_ERR_INVALID_ARG for iters
 * out of range; a wait that expires is reported by oz2_check_device_status
 * as OZ2_ERR_TIMEOUT. */
int oz2_probe_mma_rate(int64_t iters, int* cta_pairs, void* stream);

/* oz2_dgemm, oz2_dgemm_host and oz2_fallback take their workspace and
 * staging buffers from a stream-ordered memory pool that the library owns on
 * each device and that keeps freed blocks for the next call.  This returns
 * the current device's unused blocks to the system (synchronises the
 * device).  OZ2_ERR_CUDA on a CUDA failure. */
int oz2_trim_memory(void);

/* Synchronises the device and returns the device status word (OZ2_OK or
 * OZ2_ERR_TIMEOUT), clearing it. */
int oz2_check_device_status(void);

/* Human-readable name of an oz2_status. */
const char* oz2_status_string(int status);

/* ---------------------------------------------------------------------
 * Stage entry points (the same kernels the production path runs).  They
 * exist so that each stage can be checked against the CPU oracle alone.
 * ------------------------------------------------------------------- */

/* Stage 1a (Algorithm 1 "scan the exponent spans"): row max-exponents of A
 * and column max-exponents of B, non-finite detection, and the fallback
 * flags (non-finite, or max-exponent more than 128 binades from the lower
 * median of the nonzero rows).  Outputs as in oz2_ws_layout. */
int oz2_scan(int64_t m, int64_t n, int64_t k,
             const double* d_A, int64_t lda, const double* d_B, int64_t ldb,
             unsigned flags, int32_t* d_ra, int32_t* d_cb,
             uint8_t* d_row_flag, uint8_t* d_col_flag, void* stream);

/* Stage 1b+2' (§2.4, "+1" pass): magnitude planes Â_il = 2^max(-c, ⌈log2
 * |A_il|2^-ra_i⌉) (E4M3, m×k_pad and n×k_pad as the digit planes), the
 * FP8 GEMM U = ÂB̂ (exact in FP32), and the exponents d[m], e[n]
 * (oz2_scale_mode).  d_urow receives max_j U_ij.  d_mag_a/d_mag_b are outputs. */
int oz2_scale(int64_t m, int64_t n, int64_t k, int num_moduli,
              const double* d_A, int64_t lda, const double* d_B, int64_t ldb,
              const int32_t* d_ra, const int32_t* d_cb,
              const uint8_t* d_row_flag, const uint8_t* d_col_flag,
              int quant, int scale, uint8_t* d_mag_a, uint8_t* d_mag_b,
              float* d_urow, int32_t* d_d, int32_t* d_e, void* stream);

/* Stage 3 (Eq. scale and Algorithm 1 "lin:dec"): Ã = ⌊2^d_i A_il⌉ and
 * B̃ = ⌊2^e_j B_lj⌉, their centred residues, and the E4M3 digit planes in
 * the layout of oz2_plane_layout.  Rows with row_flag bit1 (columns with
 * col_flag bit1) are written as zero. */
int oz2_deconstruct(int64_t m, int64_t n, int64_t k, int num_moduli,
                    const double* d_A, int64_t lda, const double* d_B, int64_t ldb,
                    const int32_t* d_d, const int32_t* d_e,
                    const uint8_t* d_row_flag, const uint8_t* d_col_flag,
                    int quant, uint8_t* d_planes_a, uint8_t* d_planes_b,
                    void* stream);

/* Stage 4 (Eq. modgemm, Eq. sq-shortcut, Eq. kar): from digit planes in
 * the layout of oz2_plane_layout (k_pad = k rounded up to 128), the residue
 * matrices C^(i) = (A^(i) B^(i)) mod m_i, centred, as r int16 matrices,
 * each m×n column-major with leading dimension ldr ≥ m (matrix i starts at
 * element i·n·ldr; rows m..ldr-1 are not written).  Three FP8 tcgen05 MMAs
 * per modulus into two FP32 accumulators with exact accumulation (Eq.
 * accum-exact), reduced mod m_i every K-slab (32768 for square moduli, 4096
 * for nonsquare ones).  This entry has no scratch, so it never splits k
 * (oz2_dgemm_ex does for a small C with a long k; the results are the same).
 * ldr < m → OZ2_ERR_INVALID_ARG. */
int oz2_residue_gemm(int64_t m, int64_t n, int64_t k, int num_moduli,
                     const uint8_t* d_planes_a, const uint8_t* d_planes_b,
                     int16_t* d_residues, int64_t ldr, void* stream);

/* Diagnostic twin of oz2_residue_gemm on CUDA cores (same products, same
 * epilogue arithmetic, sequential k order, same output layout); slow. */
int oz2_residue_gemm_simt(int64_t m, int64_t n, int64_t k, int num_moduli,
                          const uint8_t* d_planes_a, const uint8_t* d_planes_b,
                          int16_t* d_residues, int64_t ldr, void* stream);

/* Stage 5 (Eq. garner, App. A; Algorithm 1 unscale): C_ij = RN_fp64(X_ij ·
 * 2^-(d_i+e_j)) with X_ij ∈ [-M/2, M/2) the integer whose residues are
 * C^(i)_ij.  residues: r int16 matrices, each m×n column-major with
 * leading dimension ldr ≥ m (matrix i starts at element i·n·ldr), the
 * layout oz2_residue_gemm writes; each entry any representative of its class
 * with |C^(i)_ij| < m_i (oz2_residue_gemm writes the centred one).  Entries
 * outside that range give unspecified values (never a fault). */
int oz2_reconstruct(int64_t m, int64_t n, int num_moduli,
                    const int16_t* d_residues, int64_t ldr,
                    const int32_t* d_d, const int32_t* d_e,
                    double* d_C, int64_t ldc, void* stream);

/* Stage 6 (Algorithm 1, native fallback): for every row i with row_flag
 * bit0 and every column j with col_flag bit0, C_ij = the FP64 FMA chain
 * Σ_l A_il B_lj in the order l = 0..k-1, starting from +0. */
int oz2_fallback(int64_t m, int64_t n, int64_t k,
                 const double* d_A, int64_t lda, const double* d_B, int64_t ldb,
                 const uint8_t* d_row_flag, const uint8_t* d_col_flag,
                 double* d_C, int64_t ldc, void* stream);

/* The native-FP64 comparator: C = A·B with every entry the FMA chain of
 * oz2_fallback (no emulation). */
int oz2_native_dgemm(int64_t m, int64_t n, int64_t k,
                     const double* d_A, int64_t lda, const double* d_B, int64_t ldb,
                     double* d_C, int64_t ldc, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* OZ2_H */
