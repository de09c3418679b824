// Tuned decode kernels (placeholder until the tensor-core decode lands): reports "not handled"
// so the dispatcher runs the shape-general kernel.
#include "common.cuh"

namespace fairy2i {

fairy2i_status launch_wl_decode(const void*, fairy2i_dtype, int64_t, int64_t, int64_t,
                                const uint32_t*, const float*, int64_t, int64_t, int64_t, int64_t,
                                int, float*, int64_t, cudaStream_t, bool* handled) {
  *handled = false;
  return FAIRY2I_OK;
}

}  // namespace fairy2i
