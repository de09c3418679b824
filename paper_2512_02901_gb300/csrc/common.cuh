// Shared device helpers of the Fairy2i sm_103a kernels.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "fairy2i.h"

namespace fairy2i {

// Bits latched in the per-device status word.
enum : unsigned int { kStatusNonfinite = 1u, kStatusTimeout = 2u };

// Code values: codeword i^c, c = 0:+1, 1:+i, 2:-1, 3:-i.
// PhaseQuant projection (Eq. ifairy-proj): the larger of |Re r|, |Im r| with its sign wins;
// ties |Re r| = |Im r| != 0 take the codeword counter-clockwise of the diagonal (the choice of
// k = floor(2 Arg(r)/pi + 1/2)); r = 0 gives +1. Comparisons treat -0 as +0.
__device__ __forceinline__ unsigned project_code(float a, float b) {
  const float aa = fabsf(a), ab = fabsf(b);
  if (aa > ab) return a > 0.f ? 0u : 2u;
  if (ab > aa) return b > 0.f ? 1u : 3u;
  if (aa == 0.f) return 0u;
  if (b > 0.f) return a > 0.f ? 1u : 2u;
  return a < 0.f ? 3u : 0u;
}

// Residual update of Sec. 3.3: r -= s_re b_re + i s_im b_im, one IEEE add per element.
__device__ __forceinline__ void residual_update(float& a, float& b, unsigned c, float s_re,
                                                float s_im) {
  // c even: a -= (1 - c) s_re; c odd: b -= (2 - c) s_im (selects, no branches)
  const bool odd = (c & 1u) != 0u;
  const float sg = (c & 2u) ? -1.f : 1.f;
  const float d = sg * (odd ? s_im : s_re);   // exact: a sign flip
  const float nv = __fsub_rn(odd ? b : a, d);
  a = odd ? a : nv;
  b = odd ? nv : b;
}

// Packed bit pair of a code: (Re+Im < 0, Re-Im < 0) of the codeword.
__device__ __forceinline__ unsigned neg_sum_bit(unsigned c) { return c >> 1; }            // 2,3
__device__ __forceinline__ unsigned neg_diff_bit(unsigned c) { return (c ^ (c >> 1)) & 1u; }  // 1,2

__device__ __forceinline__ void latch_status(unsigned int* status, unsigned int bit) {
  if (status) atomicOr(status, bit);
}

}  // namespace fairy2i

// Launch helpers shared by the host-side launchers.
namespace fairy2i {
inline fairy2i_status launch_status() {
  return cudaGetLastError() == cudaSuccess ? FAIRY2I_OK : FAIRY2I_ERR_CUDA;
}
// Per-device status word (defined in api.cu).
unsigned int* device_status_word();

// Raises the dynamic shared-memory limit of kernel `kern` to `bytes` on the current device, once
// per device (function attributes belong to a device's context); `done` is the caller's mask of
// devices already set (devices 0..63). Concurrent first calls set it twice, harmlessly.
template <typename Kernel>
inline bool smem_attr_once(Kernel kern, int bytes, std::atomic<uint64_t>& done) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  const uint64_t bit = uint64_t(1) << dev;
  if (done.load(std::memory_order_acquire) & bit) return true;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) !=
      cudaSuccess)
    return false;
  done.fetch_or(bit, std::memory_order_release);
  return true;
}
}  // namespace fairy2i
