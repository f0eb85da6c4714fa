// gemm_noalloc.cu -- gemm_s8s8_s32_noalloc: the exact int8 GEMM for callers
// that must not have the library allocate device memory.
//
// gemm_s8s8_s32 stages its operands (as bf16) and, for small tile counts,
// its split-K partials in a workspace the library allocates on first need.
// Some callers cannot allow that: an application whose own allocator has
// reserved nearly all device memory up front (a library-side cudaMalloc
// would fail or fragment it), a service that enforces a hard per-process
// memory budget through its own allocator and forbids hidden allocations,
// or a latency-critical loop that cannot absorb the synchronisation and
// unpredictable latency of cudaMalloc/cudaFree.  This entry point runs the
// same kernels with its scratch in a fixed, statically sized device array
// instead, and never calls an allocating routine.
#include <mutex>

#include "gb300_gemm.h"
#include "gemm_internal.h"

// Scratch of the no-allocation entry point.  Device globals are created when
// the library's device code is loaded, once per GPU, and live until the
// process exits.  In host code this name is only a host-side stand-in: the
// device address is obtained with cudaGetSymbolAddress below.
static __device__ __align__(256) uint8_t g_noalloc_scratch[GEMM_NOALLOC_SCRATCH_BYTES];

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_mu;
void *g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device, looked up on
// the first call per device and cached.  With lazy module loading (CUDA's
// default) that first lookup is also what loads this file's device code and
// so reserves the array on the device.
gemm_status_t scratch_for_current_device(void **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return GEMM_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_scratch_ptr[dev]) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return GEMM_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return GEMM_OK;
}
}  // namespace

// Forgets the cached scratch address of device `dev` (gemm_release_resources:
// after a device reset the array is created anew, at another address).
void gb300::noalloc_forget_device(int dev) {
  if (dev < 0 || dev >= kMaxDevices) return;
  std::lock_guard<std::mutex> lk(g_mu);
  g_scratch_ptr[dev] = nullptr;
}

extern "C" gemm_status_t gemm_s8s8_s32_noalloc(int64_t M, int64_t N, int64_t K, const int8_t *A,
                                               int64_t lda, const int8_t *B, int64_t ldb, int b_layout,
                                               int32_t *C, int64_t ldc, gemm_stream_t stream) {
  gemm_status_t s = gb300::validate_s8(M, N, K, A, lda, B, ldb, b_layout, C, ldc);
  if (s != GEMM_OK || M == 0 || N == 0) return s;
  void *scratch = nullptr;
  if ((s = scratch_for_current_device(&scratch)) != GEMM_OK) return s;
  return gb300::s8_gemm_into_scratch(M, N, K, A, lda, B, ldb, b_layout, C, ldc,
                                     reinterpret_cast<cudaStream_t>(stream), scratch,
                                     GEMM_NOALLOC_SCRATCH_BYTES);
}
