// The non-linear parts of a widely-linear decoder layer, for one or more tokens in the real
// layout the matmul kernels read and write ([Re | Im] halves of every vector):
//  * attention of one query over a key/value cache with Hermitian scores (Sec. 3.1,
//    Eq. hermitian-score): S[h, l] = Re(q_h^H k_{l,h}) / sqrt(d_k), softmax over l, the real
//    weights applied to the real and imaginary parts of the values separately;
//  * RMS normalisation (optionally after a residual add) and the gated activation
//    silu(gate) * up, which the widely-linear rewrite leaves real.
//
// Attention is bound by the cache reads (two floats per complex channel of every key and
// value); the arithmetic is cheap next to them, so scores and value sums are accumulated in
// two-float (compensated) form: TwoProduct by FMA and TwoSum for every product and addition,
// which keeps them accurate to a few fp32 roundings of the result whatever the cancellation.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>

#include "common.cuh"

namespace fairy2i {

namespace at {

constexpr int kThreads = 256;   // eight warps
constexpr int kWarps = kThreads / 32;
constexpr int kMaxDc = 128;     // complex channels per head (4 per lane)

// s + e holds a two-float sum; add a (exact error kept in e).
__device__ __forceinline__ void two_sum_acc(float& s, float& e, float a) {
  const float t = s + a;
  const float bp = t - s;
  e += (s - (t - bp)) + (a - bp);
  s = t;
}
// s + e += a * b with the product's rounding error kept.
__device__ __forceinline__ void two_fma_acc(float& s, float& e, float a, float b) {
  const float p = a * b;
  e += fmaf(a, b, -p);
  two_sum_acc(s, e, p);
}

// One CTA: head blockIdx.x, positions [l0, l1) of split blockIdx.y. Warp w takes positions
// l0 + w, l0 + w + 8, ...; lane j the complex channels j, j + 32, ... of the head. Online softmax
// per warp (running maximum m, sum l, two-float value sums), the eight warps combined at the end.
// Partial of the split: [m, l, Re o (dc), Im o (dc)].
__global__ void __launch_bounds__(kThreads) attn_partial_kernel(
    const float* __restrict__ q, const float* __restrict__ kc, const float* __restrict__ vc,
    int64_t L, int64_t ldkv, int64_t n, int dc, int per_split, float scale,
    float* __restrict__ part) {
  __shared__ float sm[kWarps][2 + 2 * kMaxDc];
  const int h = blockIdx.x, sp = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t l0 = (int64_t)sp * per_split, l1 = min(L, l0 + per_split);
  const int64_t c0 = (int64_t)h * dc;
  float qr[4], qi[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int c = lane + 32 * i;
    qr[i] = c < dc ? q[c0 + c] : 0.f;
    qi[i] = c < dc ? q[n + c0 + c] : 0.f;
  }
  float m = -INFINITY, lsum = 0.f;
  float orh[4] = {0.f, 0.f, 0.f, 0.f}, ore[4] = {0.f, 0.f, 0.f, 0.f};
  float oih[4] = {0.f, 0.f, 0.f, 0.f}, oie[4] = {0.f, 0.f, 0.f, 0.f};
  for (int64_t l = l0 + warp; l < l1; l += kWarps) {
    const float* kr = kc + l * ldkv + c0;
    const float* vr = vc + l * ldkv + c0;
    float s = 0.f, e = 0.f;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int c = lane + 32 * i;
      if (c < dc) {
        two_fma_acc(s, e, qr[i], kr[c]);
        two_fma_acc(s, e, qi[i], kr[n + c]);
      }
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
      const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
      const float e2 = __shfl_xor_sync(0xffffffffu, e, o);
      e += e2;
      two_sum_acc(s, e, s2);
    }
    const float score = (s + e) * scale;
    if (score > m) {   // rescale what was accumulated against the old maximum
      const float f = expf(m - score);
      lsum *= f;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        orh[i] *= f; ore[i] *= f; oih[i] *= f; oie[i] *= f;
      }
      m = score;
    }
    const float p = expf(score - m);
    lsum += p;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int c = lane + 32 * i;
      if (c < dc) {
        two_fma_acc(orh[i], ore[i], p, vr[c]);
        two_fma_acc(oih[i], oie[i], p, vr[n + c]);
      }
    }
  }
  if (lane == 0) {
    sm[warp][0] = m;
    sm[warp][1] = lsum;
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int c = lane + 32 * i;
    if (c < dc) {
      sm[warp][2 + c] = orh[i] + ore[i];
      sm[warp][2 + dc + c] = oih[i] + oie[i];
    }
  }
  __syncthreads();
  float M = -INFINITY;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) M = fmaxf(M, sm[w][0]);
  float* out = part + ((int64_t)h * gridDim.y + sp) * (2 + 2 * dc);
  for (int j = threadIdx.x; j < 2 + 2 * dc; j += kThreads) {
    float acc = 0.f, err = 0.f;
    if (j == 0) {
      acc = M;
    } else {
      for (int w = 0; w < kWarps; ++w) {
        if (sm[w][0] == -INFINITY) continue;   // a warp without positions
        two_fma_acc(acc, err, expf(sm[w][0] - M), sm[w][j]);
      }
      acc += err;
    }
    out[j] = acc;
  }
}

// Combines the splits of head blockIdx.x: o = sum_s e^(m_s - M) O_s / sum_s e^(m_s - M) l_s,
// written in the real layout (Re o at h dc + c, Im o at n + h dc + c).
__global__ void __launch_bounds__(kThreads) attn_combine_kernel(const float* __restrict__ part,
                                                                 int nsplit, int64_t n, int dc,
                                                                 float* __restrict__ out) {
  const int h = blockIdx.x;
  const float* p = part + (int64_t)h * nsplit * (2 + 2 * dc);
  float M = -INFINITY;
  for (int s = 0; s < nsplit; ++s) M = fmaxf(M, p[(int64_t)s * (2 + 2 * dc)]);
  float den = 0.f, den_e = 0.f;
  for (int s = 0; s < nsplit; ++s) {
    const float ms = p[(int64_t)s * (2 + 2 * dc)];
    if (ms != -INFINITY) two_fma_acc(den, den_e, expf(ms - M), p[(int64_t)s * (2 + 2 * dc) + 1]);
  }
  den += den_e;
  for (int j = threadIdx.x; j < 2 * dc; j += kThreads) {
    float acc = 0.f, err = 0.f;
    for (int s = 0; s < nsplit; ++s) {
      const float* ps = p + (int64_t)s * (2 + 2 * dc);
      if (ps[0] != -INFINITY) two_fma_acc(acc, err, expf(ps[0] - M), ps[2 + j]);
    }
    const float v = (acc + err) / den;
    const int c = j < dc ? j : j - dc;
    out[(j < dc ? 0 : n) + (int64_t)h * dc + c] = v;
  }
}

// One CTA per token: out = (h + delta) / sqrt(mean((h + delta)^2) + eps) * w, h_out = h + delta.
// h_out and out may alias h (each element is read before it is written, and the sums are
// complete before the first write).
__global__ void __launch_bounds__(kThreads) rmsnorm_kernel(const float* h, const float* delta,
                                                           const float* w, int64_t d, float eps,
                                                           float* h_out, float* out) {
  __shared__ float red[2][kWarps];
  const int64_t b = blockIdx.x;
  const float* hb = h + b * d;
  const float* db = delta ? delta + b * d : nullptr;
  float s = 0.f, e = 0.f;
  for (int64_t i = threadIdx.x; i < d; i += kThreads) {
    const float v = db ? hb[i] + db[i] : hb[i];
    two_fma_acc(s, e, v, v);
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
    const float e2 = __shfl_xor_sync(0xffffffffu, e, o);
    e += e2;
    two_sum_acc(s, e, s2);
  }
  if ((threadIdx.x & 31) == 0) {
    red[0][threadIdx.x >> 5] = s;
    red[1][threadIdx.x >> 5] = e;
  }
  __syncthreads();
  float ss = 0.f, se = 0.f;
#pragma unroll
  for (int wi = 0; wi < kWarps; ++wi) {
    se += red[1][wi];
    two_sum_acc(ss, se, red[0][wi]);
  }
  const float r = rsqrtf((ss + se) / (float)d + eps);
  for (int64_t i = threadIdx.x; i < d; i += kThreads) {
    const float v = db ? hb[i] + db[i] : hb[i];
    if (h_out) h_out[b * d + i] = v;
    out[b * d + i] = v * r * w[i];
  }
}

__global__ void silu_mul_kernel(const float* g, const float* u, int64_t count, float* out) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < count;
       i += (int64_t)gridDim.x * blockDim.x) {
    const float x = g[i];
    out[i] = x / (1.f + expf(-x)) * u[i];
  }
}

}  // namespace at

// Splits of the key range: about two CTAs per SM over all heads, at least 16 positions each.
static int attn_splits(int64_t L, int heads, int sms) {
  int64_t s = (2 * (int64_t)sms + heads - 1) / heads;
  s = std::min<int64_t>(s, (L + 15) / 16);
  return (int)std::max<int64_t>(1, std::min<int64_t>(s, 4096));
}

size_t attention_workspace_bytes(int64_t n, int heads, int64_t L) {
  if (n < 1 || heads < 1 || L < 1 || n % heads) return 0;
  int dev = 0, sms = 152;
  if (cudaGetDevice(&dev) == cudaSuccess) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && v > 0)
      sms = v;
  }
  const int64_t dc = n / heads;
  return (size_t)heads * attn_splits(L, heads, sms) * (2 + 2 * dc) * sizeof(float);
}

fairy2i_status launch_attention(const float* q, const float* kc, const float* vc, int64_t L,
                                int64_t ldkv, int64_t n, int heads, float* out, void* ws,
                                size_t ws_bytes, cudaStream_t stream) {
  const int64_t dc = n / heads;
  if (dc > at::kMaxDc) return FAIRY2I_ERR_INVALID_ARG;
  int dev = 0, sms = 152;
  if (cudaGetDevice(&dev) != cudaSuccess) return FAIRY2I_ERR_CUDA;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return FAIRY2I_ERR_CUDA;
  const int ns = attn_splits(L, heads, sms);
  if (ws_bytes < (size_t)heads * ns * (2 + 2 * dc) * sizeof(float)) return FAIRY2I_ERR_WORKSPACE;
  const int per = (int)((L + ns - 1) / ns);
  const float scale = 1.0f / sqrtf((float)(2 * dc));
  float* part = static_cast<float*>(ws);
  at::attn_partial_kernel<<<dim3((unsigned)heads, (unsigned)ns), at::kThreads, 0, stream>>>(
      q, kc, vc, L, ldkv, n, (int)dc, per, scale, part);
  if (cudaGetLastError() != cudaSuccess) return FAIRY2I_ERR_CUDA;
  at::attn_combine_kernel<<<(unsigned)heads, at::kThreads, 0, stream>>>(part, ns, n, (int)dc, out);
  return launch_status();
}

fairy2i_status launch_rmsnorm(const float* h, const float* delta, const float* w, int64_t B,
                              int64_t d, float eps, float* h_out, float* out, cudaStream_t stream) {
  at::rmsnorm_kernel<<<(unsigned)B, at::kThreads, 0, stream>>>(h, delta, w, d, eps, h_out, out);
  return launch_status();
}

fairy2i_status launch_silu_mul(const float* g, const float* u, int64_t count, float* out,
                               cudaStream_t stream) {
  const int64_t blocks = std::min<int64_t>((count + 255) / 256, 152 * 8);
  at::silu_mul_kernel<<<(unsigned)std::max<int64_t>(blocks, 1), 256, 0, stream>>>(g, u, count, out);
  return launch_status();
}

}  // namespace fairy2i
