// oz2_dgemm_noalloc: the emulated DGEMM for callers that cannot allocate
// device memory.
//
// Some callers may not call cudaMalloc (or cudaMallocAsync) at all: code that
// runs inside a memory-budgeted host framework whose allocator owns every
// byte of device memory, real-time or safety-reviewed loops where an
// allocation could block or fail at an unpredictable moment, and plug-ins
// that are handed only the input and output buffers.  For them this entry
// point takes its workspace from a fixed array in the library's own device
// memory instead of allocating one.
//
// The array is a file-scope `static __device__` buffer of kNoAllocScratchBytes
// bytes.  Every GPU that loads the library holds it until the process exits.
// The address host code passes to kernels is obtained with
// cudaGetSymbolAddress once per device (the array's name in host code is
// only a host-side stand-in, not a device address).
#include <mutex>

#include "oz2_common.cuh"

namespace oz2 {

// 32 MiB: room for problems up to about 512 x 512 x 512 at num_moduli = 16
// (the workspace is ~31 (m+n)·k + 24 m·n bytes at num_moduli = 12).
constexpr size_t kNoAllocScratchBytes = size_t(32) << 20;

static __device__ __align__(256) uint8_t g_noalloc_scratch[kNoAllocScratchBytes];

namespace {
struct ScratchSlot {
  bool ready = false;
  void* ptr = nullptr;
};
ScratchSlot g_slots[64];
std::mutex g_slot_mu;

// Device address of the scratch array on the current device, looked up the
// first time this device is seen.
int scratch_for_current_device(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return OZ2_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_slot_mu);
  ScratchSlot& s = g_slots[dev];
  if (!s.ready) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return OZ2_ERR_CUDA;
    s.ptr = p;
    s.ready = true;
  }
  *out = s.ptr;
  return OZ2_OK;
}
}  // namespace

}  // namespace oz2

extern "C" int oz2_dgemm_noalloc(int64_t m, int64_t n, int64_t k, const double* A, int64_t lda, const double* B,
                                 int64_t ldb, double* C, int64_t ldc, int num_moduli, void* stream) {
  if (num_moduli < 1 || num_moduli > oz2::kMaxModuli) return OZ2_ERR_UNSUPPORTED_R;
  if (m < 0 || n < 0 || k < 0) return OZ2_ERR_INVALID_ARG;
  const size_t need = (m > 0 && n > 0 && k > 0) ? oz2_workspace_size(m, n, k, num_moduli) : 0;
  if (need > oz2::kNoAllocScratchBytes) return OZ2_ERR_UNSUPPORTED;  // problem too large for the scratch array
  void* scratch = nullptr;
  if (need > 0) {
    const int st = oz2::scratch_for_current_device(&scratch);
    if (st != OZ2_OK) return st;
  }
  // The stages initialise every workspace region they read before reading it
  // (scan keys, "+1" row maxima and fallback counters are cleared on the
  // stream; planes and residues are written in full), so the previous call's
  // contents never leak into this one.
  return oz2_dgemm_ex(m, n, k, A, lda, B, ldb, C, ldc, num_moduli, OZ2_QUANT_TZ, OZ2_SCALE_R2, 0, scratch, need,
                      stream);
}
