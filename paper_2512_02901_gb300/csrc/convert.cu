// Widely-linear conversion of a real map R (2n x 2m) into the complex pair U, W
// (Sec. 3.1, Eq. UW-from-R). Elementwise and HBM-bound: 16 B read and 16 B written per
// complex position (j, k).
#include "common.cuh"

namespace fairy2i {

__device__ __forceinline__ float load_padded(const float* __restrict__ R, int64_t rows,
                                             int64_t cols, int64_t ldR, int64_t r, int64_t c) {
  return (r < rows && c < cols) ? __ldg(R + r * ldR + c) : 0.f;
}

// Thread (j, k): Re U = (R11+R22)/2, Im U = (R21-R12)/2, Re W = (R11-R22)/2,
// Im W = (R12+R21)/2 with R_ab the n x m blocks; a missing last row/column of an odd R reads 0.
__global__ void __launch_bounds__(256) convert_kernel(const float* __restrict__ R, int64_t rows,
                                                     int64_t cols, int64_t ldR, int64_t n,
                                                     int64_t m, float2* __restrict__ U,
                                                     float2* __restrict__ W, int64_t ldc) {
  const int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= m) return;
  for (int64_t j = blockIdx.y; j < n; j += gridDim.y) {
    const float r11 = load_padded(R, rows, cols, ldR, j, k);
    const float r12 = load_padded(R, rows, cols, ldR, j, m + k);
    const float r21 = load_padded(R, rows, cols, ldR, n + j, k);
    const float r22 = load_padded(R, rows, cols, ldR, n + j, m + k);
    float2 u, w;
    u.x = __fmul_rn(__fadd_rn(r11, r22), 0.5f);
    u.y = __fmul_rn(__fsub_rn(r21, r12), 0.5f);
    w.x = __fmul_rn(__fsub_rn(r11, r22), 0.5f);
    w.y = __fmul_rn(__fadd_rn(r12, r21), 0.5f);
    U[j * ldc + k] = u;
    W[j * ldc + k] = w;
  }
}

fairy2i_status launch_convert(const float* R, int64_t rows, int64_t cols, int64_t ldR, int64_t n,
                              int64_t m, float* U, float* W, int64_t ldc, cudaStream_t stream) {
  dim3 block(256);
  dim3 grid((unsigned)((m + 255) / 256), (unsigned)(n < 65535 ? n : 65535));
  convert_kernel<<<grid, block, 0, stream>>>(R, rows, cols, ldR, n, m,
                                             reinterpret_cast<float2*>(U),
                                             reinterpret_cast<float2*>(W), ldc);
  return launch_status();
}

}  // namespace fairy2i
