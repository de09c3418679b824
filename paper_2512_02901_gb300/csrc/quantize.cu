// PhaseQuant + recursive residual quantization + 2-bit packing (Sec. 3.2-3.4).
//
// Per stage t the residual R^(t) of every element is rebuilt from U or W by replaying stages
// 0..t-1 (projection + one float32 add each), so the inputs stay read-only and no residual
// buffer is needed: the replay costs O(t) float32 operations per element, while a stored
// residual would cost a write and a read of both matrices per stage. Stage t needs the two
// per-tensor sums of Eq. ifairy-scale, in float64 over a fixed tree (groups of 256 consecutive
// elements in row-major order reduced by halving strides, then the group sums the same way):
//   stage kernel: one warp per group computes its (S_re, S_im, N_re, N_im) -- the counts as
//                 integers, each S exactly in int64 when its values span at most 21 binades
//                 (then the float64 tree is exact and equals that sum), else by the float64
//                 tree; the last CTA of every 32 reduces their level-1 group, the last of
//                 those the remaining levels, and writes s = float(S / N) (0 when N = 0).
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

constexpr int kWarpsL0 = 8;                     // groups per CTA of the stage kernel
constexpr int kCtasPerL1 = kGroup / kWarpsL0;   // CTAs whose groups form one level-1 group

// Sum of the warp's 256 non-negative floats v[i] (position lane + 32 i), exact, when the nonzero
// values are normal and their exponents span at most 21 binades: every value is then an integer
// multiple of u = the ulp of the smallest one and the total is below 256 2^(emax + 1) <= 2^53 u,
// so every partial sum of the fixed tree (warp_tree256) is exact in float64 and the tree returns
// the exact sum, which int64 arithmetic gives without the float64 pipe. Returns false (and the
// caller runs the float64 tree) otherwise. Result in every lane.
__device__ __forceinline__ bool exact_sum256(const float (&v)[8], double& out) {
  uint32_t emax = 0u, emin = 255u;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint32_t b = __float_as_uint(v[i]);
    if (b != 0u) {
      emax = max(emax, b >> 23);
      emin = min(emin, b >> 23);
    }
  }
  emax = __reduce_max_sync(0xffffffffu, emax);
  emin = __reduce_min_sync(0xffffffffu, emin);
  if (emin == 255u) {   // every value is zero
    out = 0.0;
    return true;
  }
  if (emin == 0u || emax - emin > 21u) return false;
  unsigned long long sum = 0ull;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint32_t b = __float_as_uint(v[i]);
    if (b != 0u)
      sum += (unsigned long long)((b & 0x7fffffu) | 0x800000u) << ((b >> 23) - emin);
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
  // sum < 2^53 and a power of two (2^(emin - 150) >= 2^-149): both steps exact
  out = (double)sum * __longlong_as_double((long long)((int)emin - 150 + 1023) << 52);
  return true;
}

// One warp reduces level group g of `count` 4-tuples (S_re, S_im, N_re, N_im) at src, written by
// other CTAs (read through L2), with the 256-wide tree: S by the float64 tree, N (integers below
// 2^53, so every tree sum is exact) as int64. Result to dst[g] by lane 0.
__device__ void reduce_group(const double* src, int64_t count, int64_t g, double* dst, int lane) {
  double s0[8], s1[8];
  unsigned long long n0 = 0ull, n1 = 0ull;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int64_t idx = g * kGroup + lane + 32 * i;
    s0[i] = s1[i] = 0.0;
    if (idx < count) {
      s0[i] = __ldcg(src + idx * 4 + 0);
      s1[i] = __ldcg(src + idx * 4 + 1);
      n0 += (unsigned long long)__ldcg(src + idx * 4 + 2);
      n1 += (unsigned long long)__ldcg(src + idx * 4 + 3);
    }
  }
  const double S0 = warp_tree256(s0), S1 = warp_tree256(s1);
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    n0 += __shfl_xor_sync(0xffffffffu, n0, o);
    n1 += __shfl_xor_sync(0xffffffffu, n1, o);
  }
  if (lane == 0) {
    dst[g * 4 + 0] = S0;
    dst[g * 4 + 1] = S1;
    dst[g * 4 + 2] = (double)n0;
    dst[g * 4 + 3] = (double)n1;
  }
}

// Stage t of one matrix per blockIdx.y: one warp per group of 256 consecutive elements
// (row-major order) replays stages 0..t-1, projects, and writes the group's (S_re, S_im, N_re,
// N_im) to partials [2][groups][4]. The last CTA to finish among the 32 whose groups form a
// level-1 group reduces that group (lvl1 [2][nl1][4]); the last of those reduces the remaining
// levels (ping-pong through lvl [2][2][lvl_cap][4]), writes the stage-t scales and clears the
// matrix's completion counters (counters [2][nl1 + 1], zero on entry) for the next stage.
__global__ void __launch_bounds__(256, 4) quant_stage_kernel(QuantArgs q, int t, int64_t groups,
                                                          double* __restrict__ partials,
                                                          double* lvl1, double* lvl,
                                                          int64_t lvl_cap, unsigned int* counters,
                                                          float* __restrict__ scales,
                                                          unsigned int* status) {
  __shared__ int s_last;
  const int mat = blockIdx.y;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t g = (int64_t)blockIdx.x * kWarpsL0 + warp;
  const int64_t nl1 = (groups + kGroup - 1) / kGroup;
  if (g < groups) {
    const int64_t total = q.n * q.m;
    const float2* __restrict__ M = mat ? q.M[1] : q.M[0];
    float vre[8], vim[8];
    unsigned int nre = 0u, nim = 0u;
    // the eight loads of the thread are issued before any of them is used
    float2 r[8];
    {
      int64_t e = g * kGroup + lane;
      int64_t j = e / q.m, k = e - j * q.m;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        r[i] = e < total ? M[j * q.ldc + k] : make_float2(0.f, 0.f);
        e += 32;
        k += 32;
        while (k >= q.m) { k -= q.m; ++j; }
      }
    }
    bool bad = false;
    const int64_t e0 = g * kGroup + lane;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      vre[i] = vim[i] = 0.f;
      const bool live = e0 + 32 * i < total;
      unsigned c = 0u;
      if (live) {
        float a = r[i].x, b = r[i].y;
        if (t == 0) bad |= !(isfinite(a) && isfinite(b));
        c = replay(a, b, t, q.scales, mat);
        if ((c & 1u) == 0u) vre[i] = fabsf(a);
        else vim[i] = fabsf(b);
      }
      nre += __popc(__ballot_sync(0xffffffffu, live && (c & 1u) == 0u));
      nim += __popc(__ballot_sync(0xffffffffu, live && (c & 1u) != 0u));
    }
    if (bad) latch_status(status, kStatusNonfinite);
    double S_re, S_im;
    if (!exact_sum256(vre, S_re)) {
      double d[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) d[i] = (double)vre[i];
      S_re = warp_tree256(d);
    }
    if (!exact_sum256(vim, S_im)) {
      double d[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) d[i] = (double)vim[i];
      S_im = warp_tree256(d);
    }
    if (lane == 0) {
      double* p = partials + ((int64_t)mat * groups + g) * 4;
      p[0] = S_re;
      p[1] = S_im;
      p[2] = (double)nre;
      p[3] = (double)nim;
    }
  }
  // Level 1: the last of the CTAs covering level-1 group g1 reduces it.
  __syncthreads();
  unsigned int* cnt = counters + (int64_t)mat * (nl1 + 1);
  const int64_t g1 = blockIdx.x / kCtasPerL1;
  if (threadIdx.x == 0) {
    const unsigned int ctas =
        (unsigned int)min((int64_t)kCtasPerL1, (int64_t)gridDim.x - g1 * kCtasPerL1);
    __threadfence();
    s_last = atomicAdd(cnt + g1, 1u) == ctas - 1u;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  double* l1 = lvl1 + (int64_t)mat * nl1 * 4;
  if (warp == 0) reduce_group(partials + (int64_t)mat * groups * 4, groups, g1, l1, lane);
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(cnt + nl1, 1u) == (unsigned int)nl1 - 1u;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  // Levels 2 and up: this CTA, level by level.
  const double* src = l1;
  int64_t count = nl1;
  int ping = 0;
  while (count > 1) {
    const int64_t next = (count + kGroup - 1) / kGroup;
    double* dst = lvl + ((int64_t)mat * 2 + ping) * lvl_cap * 4;
    for (int64_t gg = warp; gg < next; gg += kWarpsL0) reduce_group(src, count, gg, dst, lane);
    __syncthreads();
    src = dst;
    count = next;
    ping ^= 1;
  }
  if (threadIdx.x == 0) {
    const double S_re = __ldcg(src + 0), S_im = __ldcg(src + 1);
    const double N_re = __ldcg(src + 2), N_im = __ldcg(src + 3);
    const float s_re = N_re > 0.0 ? __double2float_rn(__ddiv_rn(S_re, N_re)) : 0.f;
    const float s_im = N_im > 0.0 ? __double2float_rn(__ddiv_rn(S_im, N_im)) : 0.f;
    scales[(t * 2 + mat) * 2 + 0] = s_re;
    scales[(t * 2 + mat) * 2 + 1] = s_im;
  }
  for (int64_t i = threadIdx.x; i <= nl1; i += blockDim.x) cnt[i] = 0u;
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
  // Four word pairs per round, their loads issued before any is used (wpr is a multiple of 8).
  for (int64_t w0 = 0; w0 < wpr; w0 += 8) {
    float2 r[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t k = (w0 + 2 * u) * 16 + code_of_lane;
      r[u] = (live_row && k < q.m) ? Mrow[k] : make_float2(0.f, 0.f);
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t w = w0 + 2 * u;
      const bool live = live_row && w * 16 + code_of_lane < q.m;
      float a = r[u].x, b = r[u].y;
      for (int t = 0; t < q.T; ++t) {
        const unsigned c = project_code(a, b);
        const unsigned ns = __ballot_sync(0xffffffffu, live && neg_sum_bit(c));
        const unsigned nd = __ballot_sync(0xffffffffu, live && neg_diff_bit(c));
        if (lane < 2) {
          const uint32_t word = lane == 0 ? ((ns & 0xffffu) | (nd << 16))
                                          : ((ns >> 16) | (nd & 0xffff0000u));
          const int64_t ww = w + lane;
          const int64_t idx =
              ((((int64_t)t * 2 + mat) * tiles + j / 16) * chunks + ww / 8) * 128 +
              (j % 16) * 8 + ww % 8;
          codes[idx] = word;
        }
        residual_update(a, b, c, __ldg(q.scales + (t * 2 + mat) * 2 + 0),
                        __ldg(q.scales + (t * 2 + mat) * 2 + 1));
      }
    }
  }
}

static inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

// Workspace: partials [2][groups][4], lvl1 [2][nl1][4], lvl [2][2][lvl_cap][4] (doubles), then
// the completion counters [2][nl1 + 1] (uint32).
static void quant_layout(int64_t n, int64_t m, int64_t& groups, int64_t& nl1, int64_t& lvl_cap) {
  groups = ceil_div(n * m, kGroup);
  nl1 = ceil_div(groups, kGroup);
  lvl_cap = ceil_div(nl1, kGroup);
}

size_t quantize_workspace_bytes(int64_t n, int64_t m) {
  int64_t groups, nl1, lvl_cap;
  quant_layout(n, m, groups, nl1, lvl_cap);
  return (size_t)(2 * groups * 4 + 2 * nl1 * 4 + 2 * 2 * lvl_cap * 4) * sizeof(double) +
         (size_t)2 * (nl1 + 1) * sizeof(unsigned int);
}

fairy2i_status launch_quantize(const float* U, const float* W, int64_t n, int64_t m, int64_t ldc,
                               int T, uint32_t* codes, float* scales, void* workspace,
                               cudaStream_t stream) {
  QuantArgs q;
  q.M[0] = reinterpret_cast<const float2*>(U);
  q.M[1] = reinterpret_cast<const float2*>(W);
  q.n = n; q.m = m; q.ldc = ldc; q.T = T; q.scales = scales;
  int64_t groups, nl1, lvl_cap;
  quant_layout(n, m, groups, nl1, lvl_cap);
  double* partials = reinterpret_cast<double*>(workspace);
  double* lvl1 = partials + 2 * groups * 4;
  double* lvl = lvl1 + 2 * nl1 * 4;
  unsigned int* counters = reinterpret_cast<unsigned int*>(lvl + 2 * 2 * lvl_cap * 4);
  unsigned int* status = device_status_word();
  if (cudaMemsetAsync(counters, 0, (size_t)2 * (nl1 + 1) * sizeof(unsigned int), stream) !=
      cudaSuccess)
    return FAIRY2I_ERR_CUDA;
  for (int t = 0; t < T; ++t) {
    dim3 grid((unsigned)ceil_div(groups, kWarpsL0), 2);
    quant_stage_kernel<<<grid, 256, 0, stream>>>(q, t, groups, partials, lvl1, lvl, lvl_cap,
                                                 counters, scales, status);
    if (cudaGetLastError() != cudaSuccess) return FAIRY2I_ERR_CUDA;
  }
  const int64_t wpr = fairy2i_codes_words_per_row(m);
  const int64_t tiles = ceil_div(n, 16);
  quant_pack_kernel<<<(unsigned)ceil_div(2 * tiles * 16, 8), 256, 0, stream>>>(q, wpr, tiles, codes);
  return launch_status();
}

}  // namespace fairy2i
