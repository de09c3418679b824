// Straightforward CUDA-core evaluation of the quantized widely-linear matmul, one warp per
// complex output row. It is the fallback shape-general kernel of the decode path (any B, any
// in/out size) and the baseline the tuned kernels are measured against.
//
// A code c stores the sign bits of (Re+Im) and (Re-Im) of its codeword b = i^c; with
// sigma = sign(Re b + Im b), tau = sign(Re b - Im b):  b = ((sigma+tau) + i (sigma-tau)) / 2, so
//   s_re b_re + i s_im b_im = sigma (s_re + i s_im)/2 + tau (s_re - i s_im)/2
// (Eq. ifairy-dequant). Per (stage t, matrix M) the kernel accumulates the +-1 sums
// P = sum_k sigma_k x_k and Q = sum_k tau_k x_k (adds and subtracts only, Algorithm 1) and
// adds  h P + conj(h) Q  (U)  or  h conj(P) + conj(h) conj(Q)  (W, the conj(x) term),
// h = (s_re + i s_im)/2.
#include <cuda_bf16.h>

#include "common.cuh"

namespace fairy2i {

template <typename XT>
__device__ __forceinline__ float load_x(const XT* p);
template <>
__device__ __forceinline__ float load_x<float>(const float* p) { return __ldg(p); }
template <>
__device__ __forceinline__ float load_x<__nv_bfloat16>(const __nv_bfloat16* p) {
  return __bfloat162float(*p);
}

struct WlArgs {
  const void* x;
  int64_t B, in_features, ldx;
  const uint32_t* codes;
  const float* scales;
  int64_t n, m, out_features, wpr, ldy;
  int T;
  float* y;
};

template <typename XT, int NB>
__global__ void __launch_bounds__(256) wl_simple_kernel(WlArgs a) {
  const int lane = threadIdx.x & 31;
  const int64_t j = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int64_t b0 = (int64_t)blockIdx.y * NB;
  if (j >= a.n) return;
  const XT* __restrict__ X = reinterpret_cast<const XT*>(a.x);
  float yr[NB], yi[NB];
#pragma unroll
  for (int b = 0; b < NB; ++b) yr[b] = yi[b] = 0.f;

  for (int tm = 0; tm < 2 * a.T; ++tm) {
    // [T][2][row tile][chunk][16 rows][8 words] packing
    const int64_t tiles = (a.n + 15) / 16, chunks = a.wpr / 8;
    const uint32_t* __restrict__ row =
        a.codes + (((int64_t)tm * tiles + j / 16) * chunks) * 128 + (j % 16) * 8;
    float pr[NB], pi[NB], qr[NB], qi[NB];
#pragma unroll
    for (int b = 0; b < NB; ++b) pr[b] = pi[b] = qr[b] = qi[b] = 0.f;
    for (int64_t w = lane; w < a.wpr; w += 32) {
      const uint32_t word = __ldg(row + (w / 8) * 128 + (w % 8));
      for (int i = 0; i < 16; ++i) {
        const int64_t k = w * 16 + i;
        if (k >= a.m) break;
        const int bit = 8 * (i & 1) + (i >> 1);     // even codes in byte 0, odd in byte 1
        const uint32_t sneg = ((word >> bit) & 1u) << 31;
        const uint32_t tneg = ((word >> (16 + bit)) & 1u) << 31;
#pragma unroll
        for (int b = 0; b < NB; ++b) {
          const int64_t bb = b0 + b;
          if (bb >= a.B) break;
          const XT* xb = X + bb * a.ldx;
          const float xr = load_x<XT>(xb + k);
          const float xi = (a.m + k < a.in_features) ? load_x<XT>(xb + a.m + k) : 0.f;
          pr[b] += __uint_as_float(__float_as_uint(xr) ^ sneg);
          pi[b] += __uint_as_float(__float_as_uint(xi) ^ sneg);
          qr[b] += __uint_as_float(__float_as_uint(xr) ^ tneg);
          qi[b] += __uint_as_float(__float_as_uint(xi) ^ tneg);
        }
      }
    }
    const int t = tm >> 1, mat = tm & 1;
    const float hr = 0.5f * __ldg(a.scales + (t * 2 + mat) * 2 + 0);
    const float hi = 0.5f * __ldg(a.scales + (t * 2 + mat) * 2 + 1);
#pragma unroll
    for (int b = 0; b < NB; ++b) {
      // W multiplies conj(x): conjugate P and Q.
      const float pim = mat ? -pi[b] : pi[b];
      const float qim = mat ? -qi[b] : qi[b];
      // h P + conj(h) Q
      yr[b] += hr * pr[b] - hi * pim + hr * qr[b] + hi * qim;
      yi[b] += hr * pim + hi * pr[b] + hr * qim - hi * qr[b];
    }
  }
#pragma unroll
  for (int b = 0; b < NB; ++b) {
#pragma unroll
    for (int h = 16; h >= 1; h >>= 1) {
      yr[b] += __shfl_xor_sync(0xffffffffu, yr[b], h);
      yi[b] += __shfl_xor_sync(0xffffffffu, yi[b], h);
    }
  }
  if (lane == 0) {
#pragma unroll
    for (int b = 0; b < NB; ++b) {
      const int64_t bb = b0 + b;
      if (bb >= a.B) break;
      float* yb = a.y + bb * a.ldy;
      yb[j] = yr[b];
      if (a.n + j < a.out_features) yb[a.n + j] = yi[b];
    }
  }
}

fairy2i_status launch_wl_simple(const void* x, fairy2i_dtype xdt, int64_t B, int64_t in_features,
                                int64_t ldx, const uint32_t* codes, const float* scales,
                                int64_t n, int64_t m, int64_t out_features, int64_t wpr, int T,
                                float* y, int64_t ldy, cudaStream_t stream) {
  WlArgs a{x, B, in_features, ldx, codes, scales, n, m, out_features, wpr, ldy, T, y};
  constexpr int NB = 4;
  const int64_t chunks = (B + NB - 1) / NB;
  for (int64_t c0 = 0; c0 < chunks; c0 += 65535) {
    const int64_t c = chunks - c0 < 65535 ? chunks - c0 : 65535;
    WlArgs ac = a;
    const int64_t tok0 = c0 * NB;
    ac.B = B - tok0;
    ac.y = y + tok0 * ldy;
    if (xdt == FAIRY2I_F32) {
      ac.x = reinterpret_cast<const float*>(x) + tok0 * ldx;
      wl_simple_kernel<float, NB><<<dim3((unsigned)((n + 7) / 8), (unsigned)c), 256, 0, stream>>>(ac);
    } else {
      ac.x = reinterpret_cast<const __nv_bfloat16*>(x) + tok0 * ldx;
      wl_simple_kernel<__nv_bfloat16, NB>
          <<<dim3((unsigned)((n + 7) / 8), (unsigned)c), 256, 0, stream>>>(ac);
    }
    if (cudaGetLastError() != cudaSuccess) return FAIRY2I_ERR_CUDA;
  }
  return FAIRY2I_OK;
}

}  // namespace fairy2i
