// Phase 1's exponent scan (§2.3 Eq. scale) in pieces, for a caller whose
// operands arrive in parts while it runs: the scan keys of each part, then
// the fallback flags of an operand once all of its parts are scanned.
#pragma once

#include "oz2_common.cuh"

namespace oz2 {

// Scan keys of the rows of column-major A (m × k at A, leading dimension
// lda) and of the columns of B (k × n at B, leading dimension ldb), merged
// into out.ra and out.cb by atomic maximum, so a column chunk of A
// (A + k0·lda with k its width) merges into the same row keys as the rest.
// m or n may be 0 to scan one operand only.  The keys must be zeroed first.
cudaError_t launch_scan_keys(int64_t m, int64_t n, int64_t k, const double* A, int64_t lda, const double* B,
                             int64_t ldb, ScanOut out, cudaStream_t st);

// Fallback flags and final exponents from complete keys: A's rows when
// ops & 1, B's columns when ops & 2.  Launched as a programmatic dependent
// of the kernel before it on the stream (the scan of the operand's last
// part).
cudaError_t launch_scan_flags(int64_t m, int64_t n, int ops, unsigned flags, ScanOut out, Oz2Device* dev,
                              cudaStream_t st);

}  // namespace oz2
