// PhaseQuant + recursive residual quantization + 2-bit packing (Sec. 3.2-3.4).
//
// Per stage t the residual R^(t) of every element is rebuilt from U or W by replaying stages
// 0..t-1 (projection + one float32 add each), so the inputs stay read-only and no residual
// buffer is needed. Stage t then needs the two per-tensor sums of Eq. ifairy-scale:
//   level-0 kernel: one warp per group of 256 consecutive elements (row-major order), the
//                   four float64 quantities (S_re, S_im, N_re, N_im) reduced by the fixed
//                   stride-halving tree;
//   reduce kernel:  one CTA per matrix reduces the group sums with the same tree, level by
//                   level, and writes s = float(S / N) (0 when N = 0).
// After the T stages a pack kernel replays all stages once more and writes the 2-bit codes
// with warp ballots (32 consecutive codes -> two words).
#include "common.cuh"

namespace fairy2i {

constexpr int kGroup = 256;

struct QuantArgs {
  const float2* M[2];  // U, W
  int64_t n, m, ldc;
  int T;
  const float* scales;  // [T][2][2]
};

// Warp-level fixed tree over 256 values held as v[i] = value at position lane + 32 i:
// h = 128, 64, 32 pair registers within a thread, h = 16..1 pair lanes. Result in lane 0.
__device__ __forceinline__ double warp_tree256(double v[8]) {
#pragma unroll
  for (int i = 0; i < 4; ++i) v[i] = __dadd_rn(v[i], v[i + 4]);
#pragma unroll
  for (int i = 0; i < 2; ++i) v[i] = __dadd_rn(v[i], v[i + 2]);
  double s = __dadd_rn(v[0], v[1]);
#pragma unroll
  for (int h = 16; h >= 1; h >>= 1) s = __dadd_rn(s, __shfl_down_sync(0xffffffffu, s, h));
  return s;
}

// Replays stages 0..t-1 on (a, b) and returns the stage-t code.
__device__ __forceinline__ unsigned replay(float& a, float& b, int t, const float* __restrict__ sc,
                                           int mat) {
  for (int s = 0; s < t; ++s) {
    const unsigned c = project_code(a, b);
    residual_update(a, b, c, __ldg(sc + (s * 2 + mat) * 2 + 0), __ldg(sc + (s * 2 + mat) * 2 + 1));
  }
  return project_code(a, b);
}

// partials: [2][groups][4] doubles (S_re, S_im, N_re, N_im) of stage t.
__global__ void __launch_bounds__(256) quant_level0_kernel(QuantArgs q, int t, int64_t groups,
                                                           double* __restrict__ partials,
                                                           unsigned int* status) {
  const int mat = blockIdx.y;
  const int lane = threadIdx.x & 31;
  const int64_t g = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  if (g >= groups) return;
  const int64_t total = q.n * q.m;
  const float2* __restrict__ M = mat ? q.M[1] : q.M[0];
  double sre[8], sim[8], nre[8], nim[8];
  int64_t e = g * kGroup + lane;
  int64_t j = e / q.m, k = e - j * q.m;
  bool bad = false;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    sre[i] = sim[i] = nre[i] = nim[i] = 0.0;
    if (e < total) {
      const float2 r = M[j * q.ldc + k];
      float a = r.x, b = r.y;
      if (t == 0) bad |= !(isfinite(a) && isfinite(b));
      const unsigned c = replay(a, b, t, q.scales, mat);
      if ((c & 1u) == 0u) { sre[i] = (double)fabsf(a); nre[i] = 1.0; }
      else { sim[i] = (double)fabsf(b); nim[i] = 1.0; }
    }
    e += 32;
    k += 32;
    while (k >= q.m) { k -= q.m; ++j; }
  }
  if (bad) latch_status(status, kStatusNonfinite);
  const double S_re = warp_tree256(sre);
  const double S_im = warp_tree256(sim);
  const double N_re = warp_tree256(nre);
  const double N_im = warp_tree256(nim);
  if (lane == 0) {
    double* p = partials + ((int64_t)mat * groups + g) * 4;
    p[0] = S_re; p[1] = S_im; p[2] = N_re; p[3] = N_im;
  }
}

// One CTA per matrix: reduce `groups` 4-tuples to one with the same 256-wide tree, level by
// level (ping-pong through lvl[2]), then write the stage-t scales.
__global__ void __launch_bounds__(512) quant_reduce_kernel(const double* partials,
                                                            int64_t groups, double* lvl,
                                                            int64_t lvl_cap, int t,
                                                            float* __restrict__ scales) {
  const int mat = blockIdx.x;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  const double* src = partials + (int64_t)mat * groups * 4;
  double* bufs[2] = {lvl + ((int64_t)mat * 2 + 0) * lvl_cap * 4,
                     lvl + ((int64_t)mat * 2 + 1) * lvl_cap * 4};
  int64_t count = groups;
  int ping = 0;
  while (count > 1) {
    const int64_t next = (count + kGroup - 1) / kGroup;
    double* dst = bufs[ping];
    for (int64_t g = warp; g < next; g += nwarps) {
      double v[4][8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int64_t idx = g * kGroup + lane + 32 * i;
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4) v[q4][i] = idx < count ? src[idx * 4 + q4] : 0.0;
      }
      double r[4];
#pragma unroll
      for (int q4 = 0; q4 < 4; ++q4) r[q4] = warp_tree256(v[q4]);
      if (lane == 0) {
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4) dst[g * 4 + q4] = r[q4];
      }
    }
    __syncthreads();
    src = dst;
    count = next;
    ping ^= 1;
  }
  if (threadIdx.x == 0) {
    const double S_re = src[0], S_im = src[1], N_re = src[2], N_im = src[3];
    const float s_re = N_re > 0.0 ? __double2float_rn(__ddiv_rn(S_re, N_re)) : 0.f;
    const float s_im = N_im > 0.0 ? __double2float_rn(__ddiv_rn(S_im, N_im)) : 0.f;
    scales[(t * 2 + mat) * 2 + 0] = s_re;
    scales[(t * 2 + mat) * 2 + 1] = s_im;
  }
}

// One warp per (matrix, row) of the padded row range (16 rows per tile); 32 consecutive codes
// per iteration -> ballots -> two words per stage: word0 = (neg_sum lanes 0-15) |
// (neg_diff lanes 0-15) << 16, word1 likewise for lanes 16-31, with the lanes permuted so
// that each ballot bit lands at its code's bit. Words are stored in
// [T][2][row tile][chunk of 8 words][16 rows][8 words] order; rows >= n are written as 0.
__global__ void __launch_bounds__(256) quant_pack_kernel(QuantArgs q, int64_t wpr, int64_t tiles,
                                                         uint32_t* __restrict__ codes) {
  const int lane = threadIdx.x & 31;
  const int64_t rows = tiles * 16;
  const int64_t row = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  if (row >= 2 * rows) return;
  const int mat = (int)(row / rows);
  const int64_t j = row - (int64_t)mat * rows;
  const bool live_row = j < q.n;
  const float2* __restrict__ Mrow = (mat ? q.M[1] : q.M[0]) + (live_row ? j : 0) * q.ldc;
  const int64_t chunks = wpr / 8;
  // Lane l handles code i = 2 (l % 8) + (l / 8) % 2 of word w + l / 16, so that the ballot bit
  // of lane l is bit 8 (i % 2) + i / 2 of the word (even codes in byte 0, odd codes in byte 1).
  const int code_of_lane = (lane >> 4) * 16 + 2 * (lane & 7) + ((lane >> 3) & 1);
  for (int64_t w = 0; w < wpr; w += 2) {
    const int64_t k = w * 16 + code_of_lane;
    float a = 0.f, b = 0.f;
    const bool live = live_row && k < q.m;
    if (live) { const float2 r = Mrow[k]; a = r.x; b = r.y; }
    for (int t = 0; t < q.T; ++t) {
      const unsigned c = project_code(a, b);
      const unsigned ns = __ballot_sync(0xffffffffu, live && neg_sum_bit(c));
      const unsigned nd = __ballot_sync(0xffffffffu, live && neg_diff_bit(c));
      if (lane < 2) {
        const uint32_t word = lane == 0 ? ((ns & 0xffffu) | (nd << 16))
                                        : ((ns >> 16) | (nd & 0xffff0000u));
        const int64_t ww = w + lane;
        const int64_t idx = ((((int64_t)t * 2 + mat) * tiles + j / 16) * chunks + ww / 8) * 128 +
                            (j % 16) * 8 + ww % 8;
        codes[idx] = word;
      }
      residual_update(a, b, c, __ldg(q.scales + (t * 2 + mat) * 2 + 0),
                      __ldg(q.scales + (t * 2 + mat) * 2 + 1));
    }
  }
}

static inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

size_t quantize_workspace_bytes(int64_t n, int64_t m) {
  const int64_t groups = ceil_div(n * m, kGroup);
  const int64_t lvl_cap = ceil_div(groups, kGroup);
  return (size_t)(2 * groups * 4 + 2 * 2 * lvl_cap * 4) * sizeof(double);
}

fairy2i_status launch_quantize(const float* U, const float* W, int64_t n, int64_t m, int64_t ldc,
                               int T, uint32_t* codes, float* scales, void* workspace,
                               cudaStream_t stream) {
  QuantArgs q;
  q.M[0] = reinterpret_cast<const float2*>(U);
  q.M[1] = reinterpret_cast<const float2*>(W);
  q.n = n; q.m = m; q.ldc = ldc; q.T = T; q.scales = scales;
  const int64_t groups = ceil_div(n * m, kGroup);
  const int64_t lvl_cap = ceil_div(groups, kGroup);
  double* partials = reinterpret_cast<double*>(workspace);
  double* lvl = partials + 2 * groups * 4;
  unsigned int* status = device_status_word();
  for (int t = 0; t < T; ++t) {
    dim3 grid((unsigned)ceil_div(groups, 8), 2);
    quant_level0_kernel<<<grid, 256, 0, stream>>>(q, t, groups, partials, status);
    if (cudaGetLastError() != cudaSuccess) return FAIRY2I_ERR_CUDA;
    quant_reduce_kernel<<<2, 512, 0, stream>>>(partials, groups, lvl, lvl_cap, t, scales);
    if (cudaGetLastError() != cudaSuccess) return FAIRY2I_ERR_CUDA;
  }
  const int64_t wpr = fairy2i_codes_words_per_row(m);
  const int64_t tiles = ceil_div(n, 16);
  quant_pack_kernel<<<(unsigned)ceil_div(2 * tiles * 16, 8), 256, 0, stream>>>(q, wpr, tiles, codes);
  return launch_status();
}

}  // namespace fairy2i
