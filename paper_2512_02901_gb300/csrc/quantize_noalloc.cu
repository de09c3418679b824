// fairy2i_quantize_noalloc: the quantizer with its scratch in a fixed device array, for
// callers that may not allocate device memory themselves.
//
// The quantizer needs scratch for its per-group partial sums. fairy2i_quantize takes that
// scratch from the caller; this variant takes it from `g_noalloc_scratch`, a file-scope
// __device__ array that every device which loads the library holds until the process exits.
// The host never uses the array's name as an address (on the host it is only a stand-in); the
// device address is looked up with cudaGetSymbolAddress once per device, with that device
// current, on the first call made on it.
#include <cuda_runtime.h>

#include <mutex>

#include "common.cuh"

namespace fairy2i {

size_t quantize_workspace_bytes(int64_t n, int64_t m);
fairy2i_status launch_quantize(const float* U, const float* W, int64_t n, int64_t m, int64_t ldc,
                               int T, uint32_t* codes, float* scales, void* workspace,
                               cudaStream_t stream);

static __device__ __align__(256) unsigned char g_noalloc_scratch[FAIRY2I_NOALLOC_SCRATCH_BYTES];

static void* g_noalloc_ptr[64];
static std::mutex g_noalloc_mu;

// Device address of the scratch array for the current device (looked up once per device).
static fairy2i_status noalloc_scratch(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return FAIRY2I_ERR_CUDA;
  if (dev < 0 || dev >= 64) return FAIRY2I_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) {
      cudaGetLastError();
      return FAIRY2I_ERR_CUDA;
    }
    g_noalloc_ptr[dev] = p;
  }
  *out = g_noalloc_ptr[dev];
  return FAIRY2I_OK;
}

}  // namespace fairy2i

extern "C" fairy2i_status fairy2i_quantize_noalloc(const float* U, const float* W, int64_t n,
                                                   int64_t m, int64_t ldc, int T, uint32_t* codes,
                                                   float* scales, void* stream) {
  using namespace fairy2i;
  if (!U || !W || !codes || !scales || n < 1 || m < 1 || T < 1 || T > FAIRY2I_MAX_STAGES)
    return FAIRY2I_ERR_INVALID_ARG;
  if (n > (int64_t(1) << 40) / m || ldc < m) return FAIRY2I_ERR_SHAPE;
  if ((reinterpret_cast<uintptr_t>(U) & 7) || (reinterpret_cast<uintptr_t>(W) & 7) ||
      (reinterpret_cast<uintptr_t>(codes) & 15) || (reinterpret_cast<uintptr_t>(scales) & 3))
    return FAIRY2I_ERR_ALIGNMENT;
  if (quantize_workspace_bytes(n, m) > (size_t)FAIRY2I_NOALLOC_SCRATCH_BYTES)
    return FAIRY2I_ERR_WORKSPACE;
  void* scratch = nullptr;
  fairy2i_status st = noalloc_scratch(&scratch);
  if (st != FAIRY2I_OK) return st;
  // Every entry of the scratch that a kernel reads was written earlier in the same call, so
  // nothing left by a previous call needs clearing.
  return launch_quantize(U, W, n, m, ldc, T, codes, scales, scratch,
                         static_cast<cudaStream_t>(stream));
}
