// Gradients of the quantized widely-linear layer for quantization-aware training (Sec. 3.2 QAT
// paragraph, Sec. 3.3 QAT): the straight-through weight gradient and the gradient that flows
// through the per-tensor scales of the residual stages.
//
// Weight gradient. For y = U^ x + W^ conj(x) and the output gradient g, the gradients of the
// dequantized matrices are dU = sum_b g_b conj(x_b)^T and dW = sum_b g_b x_b^T. Both come from
// the four real cross products G11 = sum g_re x_re^T, G12 = sum g_re x_im^T, G21 = sum g_im x_re^T,
// G22 = sum g_im x_im^T: dU = (G11 + G22) + i (G21 - G12), dW = (G11 - G22) + i (G12 + G21),
// i.e. one real GEMM G = g~^T x~ (2n x B times B x 2m) serves both -- two real products per
// complex product, fewer than the three of Gauss's trick, which saves a product only when a
// single complex product is wanted. The GEMM runs on the 5th-generation tensor cores: bf16 x and
// g are first transposed to token-contiguous rows; a CTA computes one 64 x 64 block of dU and dW
// as a 128 x 128 tile D = [g_re ; g_im rows] x [x_re ; x_im rows]^T (tcgen05.mma kind::f16, A and
// B in shared memory by TMA with 128-byte swizzle, f32 accumulate in tensor memory), and the
// epilogue combines the four 64 x 64 quadrants.
//
// Scale path. With the codes held fixed the loss is linear in the scales; backpropagating through
// r^(t+1) = r^(t) - (s_re b_re + i s_im b_im), s_re = mean over the +-1 codes of |Re r^(t)|:
//   s^_t = <dM - r^_(t+1), b^t> (real part over the +-1 codes, imaginary over the +-i codes),
//   r^_t = r^_(t+1) + s^_re,t sign(Re r^(t)) [+-1 code] / N_re + i s^_im,t sign(Im r^(t)) [+-i] / N_im,
// from r^_T = 0, over t = T-1 .. 0; r^_0 is the master gradient through the scales. Every sum is
// float64 in a fixed order; r^(t) is replayed from the master in float32 exactly as the quantizer
// computes it.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <mutex>

#include "common.cuh"
#include "ptx.cuh"
#include "tc.cuh"

namespace fairy2i {

namespace gr {

constexpr int kThreads = 192;      // warp 0: TMA, warp 1: MMA, warps 2-5: epilogue
constexpr int kStages = 4;
constexpr int kTile = 16 * 1024;   // 128 rows x 128 B (64 bf16 of K), 128-byte swizzle
constexpr int kStage = 2 * kTile;  // A and B
constexpr int kOffBar = kStages * kStage;
constexpr int kSmemBytes = kOffBar + 256 + 1024;
constexpr uint64_t kWaitNs = 1000000000ull;
// kind::f16, bf16 A and B, f32 D, K-major, N = 128, M = 128.
constexpr uint32_t kIdesc =
    (1u << 4) | (1u << 7) | (1u << 10) | ((128u >> 3) << 17) | ((128u >> 4) << 24);

__device__ __forceinline__ uint64_t desc_sw128(uint32_t addr) {
  return (uint64_t)((addr >> 4) & 0x3FFFu) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
         (1ull << 46) | (2ull << 61);
}
// D[tmem] (+)= A[smem] B[smem]^T, bf16, f32 accumulate.
__device__ __forceinline__ void mma_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                       uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %3, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %4, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(accumulate), "r"(kIdesc)
      : "memory");
}
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* v) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
      "%11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, "
      "%29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Token-contiguous copy of the two halves of a real-layout activation: out[f][b] for feature f of
// part p at row p rows_half + f (rows_half = ceil(features / 2); the odd last Im row is zero),
// tokens b < Bpad (zero beyond B). 32 x 32 tiles through shared memory.
__global__ void transpose_kernel(const __nv_bfloat16* __restrict__ in, int64_t ld, int64_t B,
                                 int64_t features, int64_t half, int64_t Bpad,
                                 __nv_bfloat16* __restrict__ out) {
  __shared__ unsigned short t[32][33];
  const int64_t r0 = (int64_t)blockIdx.y * 32, b0 = (int64_t)blockIdx.x * 32;   // rows of out
  const int tx = threadIdx.x, ty = threadIdx.y;                                 // 32 x 8
  for (int i = ty; i < 32; i += 8) {
    const int64_t b = b0 + i, r = r0 + tx;
    unsigned short v = 0;
    if (b < B && r < 2 * half) {
      const int64_t f = r < half ? r : (r - half) + half;   // feature index in the token row
      const bool real_row = r < half || (r - half) + half < features;
      if (real_row && f < features) v = __bfloat16_as_ushort(in[b * ld + f]);
    }
    t[i][tx] = v;
  }
  __syncthreads();
  for (int i = ty; i < 32; i += 8) {
    const int64_t r = r0 + i, b = b0 + tx;
    if (r < 2 * half && b < Bpad) out[r * Bpad + b] = __ushort_as_bfloat16(t[tx][i]);
  }
}

struct GArgs {
  float* dU;
  float* dW;
  unsigned int* status;
  int64_t n, m, ldc;
  int ksteps;      // Bpad / 64
  int kblocks;     // ceil(m / 64)
  int accumulate;
};

__device__ __forceinline__ bool wait_b(uint64_t* bar, uint32_t parity, volatile int* abort,
                                       unsigned int* status) {
  if (*abort) return false;
  if (mbar_wait_spin(bar, parity, kWaitNs)) return true;
  *abort = 1;
  latch_status(status, kStatusTimeout);
  return false;
}

// One CTA: output block (j0 = 64 blockIdx.y, k0 = 64 blockIdx.x) of dU and dW.
__global__ void __launch_bounds__(kThreads, 1) ste_gemm_kernel(
    const GArgs a, const __grid_constant__ CUtensorMap gmap, const __grid_constant__ CUtensorMap xmap) {
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = align_smem_1024(smem_raw);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kOffBar);
  uint64_t* empty = full + kStages;
  uint64_t* done = empty + kStages;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(done + 1);
  volatile int* abort_flag = reinterpret_cast<int*>(tslot + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t j0 = (int64_t)blockIdx.y * 64, k0 = (int64_t)blockIdx.x * 64;
  if (warp == 0) {
    if (lane < kStages) {
      mbar_init(&full[lane], 1);
      mbar_init(&empty[lane], 1);
    }
    if (lane == 0) {
      mbar_init(done, 1);
      *abort_flag = 0;
    }
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(tslot, 128);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;
  pdl_launch_dependents();
  if (warp == 0) {
    if (lane == 0) {
      prefetch_tensormap(&gmap);
      prefetch_tensormap(&xmap);
      pdl_wait_primary();
      int issued = 0;
      for (int ks = 0; ks < a.ksteps; ++ks) {
        const int st = ks % kStages;
        if (ks >= kStages && !wait_b(&empty[st], ((ks / kStages) - 1) & 1, abort_flag, a.status))
          break;
        issued = ks + 1;
        mbar_arrive_expect_tx(&full[st], (uint32_t)kStage);
        unsigned char* sa = smem + st * kStage;
        // A rows 0-63: g_re of rows j0..; 64-127: g_im (gT row n + j); B likewise from xT
        tma_load_2d(sa, &gmap, ks * 64, (int32_t)j0, &full[st]);
        tma_load_2d(sa + kTile / 2, &gmap, ks * 64, (int32_t)(a.n + j0), &full[st]);
        tma_load_2d(sa + kTile, &xmap, ks * 64, (int32_t)k0, &full[st]);
        tma_load_2d(sa + kTile + kTile / 2, &xmap, ks * 64, (int32_t)(a.m + k0), &full[st]);
      }
      // every copy lands before the CTA exits
      for (int q = max(0, issued - kStages); q < issued; ++q)
        (void)mbar_wait_timed(&full[q % kStages], (q / kStages) & 1, kWaitNs);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = true;
      for (int ks = 0; ks < a.ksteps; ++ks) {
        const int st = ks % kStages;
        ok = wait_b(&full[st], (ks / kStages) & 1, abort_flag, a.status);
        if (!ok) break;
        tc_fence_after();
        const uint32_t sa = smem_u32(smem + st * kStage);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)   // K = 16 per MMA: 32 bytes of each 128-byte row
          mma_ss(tmem, desc_sw128(sa + kk * 32), desc_sw128(sa + kTile + kk * 32),
                 (ks > 0 || kk > 0) ? 1u : 0u);
        mma_commit(&empty[st]);
      }
      mma_commit(done);   // also after an abort: the MMAs issued finish before TMEM is freed
    }
    __syncwarp();
  } else {
    // ---- epilogue: lane r of D holds g_re row j0 + r (r < 64) or g_im row j0 + r - 64 ----
    const int q = warp & 3;                  // TMEM lane quarter of this warp
    const int r = q * 32 + lane;             // D row
    const bool ok = wait_b(done, 0, abort_flag, a.status) || false;
    tc_fence_after();
    float* stage = reinterpret_cast<float*>(smem);   // [64 rows][128 floats]: G21 | G22
    float v[128];
    if (ok) {
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(tmem + ((uint32_t)(q * 32) << 16) + c * 32, v + 32 * c);
      tmem_wait_ld();
    }
    if (r >= 64) {
#pragma unroll
      for (int c = 0; c < 128; ++c) stage[(r - 64) * 129 + c] = ok ? v[c] : 0.f;
    }
    asm volatile("bar.sync 1, 128;" ::: "memory");
    if (r < 64 && ok && !*abort_flag) {
      const int64_t j = j0 + r;
      if (j < a.n) {
        const float* o = stage + r * 129;
        float2* du = reinterpret_cast<float2*>(a.dU + 2 * (j * a.ldc));
        float2* dw = reinterpret_cast<float2*>(a.dW + 2 * (j * a.ldc));
#pragma unroll
        for (int c = 0; c < 64; ++c) {
          const int64_t k = k0 + c;
          if (k >= a.m) continue;
          // v: G11 (cols 0-63), G12 (64-127); o: G21, G22
          float2 u = make_float2(v[c] + o[64 + c], o[c] - v[64 + c]);
          float2 w = make_float2(v[c] - o[64 + c], v[64 + c] + o[c]);
          if (a.accumulate) {
            const float2 u0 = du[k], w0 = dw[k];
            u.x += u0.x; u.y += u0.y; w.x += w0.x; w.y += w0.y;
          }
          du[k] = u;
          dw[k] = w;
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 128);
}

// ---------------------------------------------------------------- scale path
constexpr int kRedBlocks = 296;    // partial sums of the reductions (fixed, so the order is too)
constexpr int kRedThreads = 256;

// Code of element (j, k) of matrix M at stage t from the packed layout.
__device__ __forceinline__ unsigned code_at(const uint32_t* codes, int64_t row_tiles, int64_t wpr,
                                            int t, int M, int64_t j, int64_t k) {
  const int64_t w = k >> 4, i = k & 15;
  const int64_t idx = ((((int64_t)(t * 2 + M) * row_tiles + (j >> 4)) * (wpr >> 3) + (w >> 3)) *
                           16 + (j & 15)) * 8 + (w & 7);
  const uint32_t word = codes[idx];
  const int b = 8 * (int)(i & 1) + (int)(i >> 1);
  const unsigned ns = (word >> b) & 1u, nd = (word >> (16 + b)) & 1u;
  return ns == 0 ? nd : 3u - nd;   // (0,0) +1, (0,1) +i, (1,1) -1, (1,0) -i
}

// Per-block float64 partial sums, for stage t of both matrices: <dM - r^, b^t> re and im parts,
// and the code counts of the two sets. part[blk][M][4].
__global__ void __launch_bounds__(kRedThreads) scale_reduce_kernel(
    const float* __restrict__ dU, const float* __restrict__ dW, int64_t ldg,
    const float* __restrict__ rU, const float* __restrict__ rW, int64_t ldr,
    const uint32_t* __restrict__ codes, int64_t n, int64_t m, int64_t row_tiles, int64_t wpr, int t,
    double* __restrict__ part) {
  __shared__ double sh[kRedThreads / 32][8];
  double acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  const int64_t total = n * m;
  for (int64_t e = (int64_t)blockIdx.x * kRedThreads + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * kRedThreads) {
    const int64_t j = e / m, k = e - j * m;
#pragma unroll
    for (int M = 0; M < 2; ++M) {
      const float* d = M ? dW : dU;
      const float* rh = M ? rW : rU;
      const unsigned c = code_at(codes, row_tiles, wpr, t, M, j, k);
      const double gre = (double)d[2 * (j * ldg + k)] - (double)rh[2 * (j * ldr + k)];
      const double gim = (double)d[2 * (j * ldg + k) + 1] - (double)rh[2 * (j * ldr + k) + 1];
      if (c == 0u || c == 2u) {
        acc[M * 4 + 0] += c == 0u ? gre : -gre;
        acc[M * 4 + 2] += 1.0;
      } else {
        acc[M * 4 + 1] += c == 1u ? gim : -gim;
        acc[M * 4 + 3] += 1.0;
      }
    }
  }
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) acc[i] += __shfl_xor_sync(0xffffffffu, acc[i], o);
  if ((threadIdx.x & 31) == 0)
#pragma unroll
    for (int i = 0; i < 8; ++i) sh[threadIdx.x >> 5][i] = acc[i];
  __syncthreads();
  if (threadIdx.x < 8) {
    double s = 0.0;
    for (int w = 0; w < kRedThreads / 32; ++w) s += sh[w][threadIdx.x];
    part[blockIdx.x * 8 + threadIdx.x] = s;
  }
}

// r^ += s^_re sign(Re r^(t)) [+-1 code] / N_re + i s^_im sign(Im r^(t)) [+-i code] / N_im for both
// matrices, with s^ and N summed from the partials in block order (every thread the same sum);
// thread 0 of block 0 writes s^ of stage t.
__global__ void __launch_bounds__(kRedThreads) scale_update_kernel(
    const float* __restrict__ U, const float* __restrict__ W, int64_t ldm, const float* scales,
    const uint32_t* __restrict__ codes, int64_t n, int64_t m, int64_t row_tiles, int64_t wpr, int t,
    const double* __restrict__ part, int nblk, float* rU, float* rW, int64_t ldr, float* shat) {
  __shared__ double tot[8];
  if (threadIdx.x < 8) {
    double s = 0.0;
    for (int b = 0; b < nblk; ++b) s += part[b * 8 + threadIdx.x];
    tot[threadIdx.x] = s;
  }
  __syncthreads();
  if (blockIdx.x == 0 && threadIdx.x < 4) {
    const int M = threadIdx.x >> 1, p = threadIdx.x & 1;
    shat[(t * 2 + M) * 2 + p] = (float)tot[M * 4 + p];
  }
  const int64_t total = n * m;
  for (int64_t e = (int64_t)blockIdx.x * kRedThreads + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * kRedThreads) {
    const int64_t j = e / m, k = e - j * m;
#pragma unroll
    for (int M = 0; M < 2; ++M) {
      const float* src = M ? W : U;
      float re = src[2 * (j * ldm + k)], im = src[2 * (j * ldm + k) + 1];
      for (int tt = 0; tt < t; ++tt) {
        const unsigned cc = code_at(codes, row_tiles, wpr, tt, M, j, k);
        residual_update(re, im, cc, scales[(tt * 2 + M) * 2], scales[(tt * 2 + M) * 2 + 1]);
      }
      const unsigned c = code_at(codes, row_tiles, wpr, t, M, j, k);
      float* rh = M ? rW : rU;
      if (c == 0u || c == 2u) {
        const double nre = tot[M * 4 + 2];
        const double sg = re > 0.f ? 1.0 : (re < 0.f ? -1.0 : 0.0);
        rh[2 * (j * ldr + k)] += (float)(tot[M * 4 + 0] * sg / nre);
      } else {
        const double nim = tot[M * 4 + 3];
        const double sg = im > 0.f ? 1.0 : (im < 0.f ? -1.0 : 0.0);
        rh[2 * (j * ldr + k) + 1] += (float)(tot[M * 4 + 1] * sg / nim);
      }
    }
  }
}

__global__ void zero_kernel(float* p, int64_t rows, int64_t cols, int64_t ld) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < rows * cols;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = e / cols, c = e - r * cols;
    p[r * ld + c] = 0.f;
  }
}

}  // namespace gr

namespace {
std::mutex g_gr_mu;
PFN_cuTensorMapEncodeTiled_v12000 g_gr_encode = nullptr;
}  // namespace

static PFN_cuTensorMapEncodeTiled_v12000 gr_encoder() {
  std::lock_guard<std::mutex> lock(g_gr_mu);
  if (!g_gr_encode) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return nullptr;
    g_gr_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  return g_gr_encode;
}

static int64_t pad64(int64_t v) { return (v + 63) / 64 * 64; }

size_t ste_grad_workspace_bytes(int64_t B, int64_t in_features, int64_t out_features) {
  const int64_t n = (out_features + 1) / 2, m = (in_features + 1) / 2;
  const int64_t Bp = pad64(B);
  return (size_t)(2 * n + 2 * m) * Bp * 2 + 256;
}

fairy2i_status launch_ste_grad(const void* x, int64_t ldx, const void* g, int64_t ldg, int64_t B,
                               int64_t in_features, int64_t out_features, float* dU, float* dW,
                               int64_t ldc, int accumulate, void* ws, cudaStream_t stream) {
  using namespace gr;
  const int64_t n = (out_features + 1) / 2, m = (in_features + 1) / 2;
  const int64_t Bp = pad64(B);
  __nv_bfloat16* gT = static_cast<__nv_bfloat16*>(ws);
  __nv_bfloat16* xT = gT + 2 * n * Bp;
  const dim3 tb(32, 8);
  transpose_kernel<<<dim3((unsigned)(Bp / 32), (unsigned)((2 * n + 31) / 32)), tb, 0, stream>>>(
      static_cast<const __nv_bfloat16*>(g), ldg, B, out_features, n, Bp, gT);
  transpose_kernel<<<dim3((unsigned)(Bp / 32), (unsigned)((2 * m + 31) / 32)), tb, 0, stream>>>(
      static_cast<const __nv_bfloat16*>(x), ldx, B, in_features, m, Bp, xT);
  if (cudaGetLastError() != cudaSuccess) return FAIRY2I_ERR_CUDA;
  PFN_cuTensorMapEncodeTiled_v12000 enc = gr_encoder();
  if (!enc) return FAIRY2I_ERR_CUDA;
  CUtensorMap gmap, xmap;
  const cuuint32_t box[2] = {64, 64};
  const cuuint32_t estr[2] = {1, 1};
  {
    const cuuint64_t dims[2] = {(cuuint64_t)Bp, (cuuint64_t)(2 * n)};
    const cuuint64_t strides[1] = {(cuuint64_t)Bp * 2};
    if (enc(&gmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, gT, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return FAIRY2I_ERR_CUDA;
  }
  {
    const cuuint64_t dims[2] = {(cuuint64_t)Bp, (cuuint64_t)(2 * m)};
    const cuuint64_t strides[1] = {(cuuint64_t)Bp * 2};
    if (enc(&xmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, xT, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return FAIRY2I_ERR_CUDA;
  }
  GArgs a;
  a.dU = dU;
  a.dW = dW;
  a.status = device_status_word();
  a.n = n;
  a.m = m;
  a.ldc = ldc;
  a.ksteps = (int)(Bp / 64);
  a.kblocks = (int)((m + 63) / 64);
  a.accumulate = accumulate;
  auto kern = ste_gemm_kernel;
  static std::atomic<uint64_t> smem_set{0};
  if (!smem_attr_once(kern, kSmemBytes, smem_set)) return FAIRY2I_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)a.kblocks, (unsigned)((n + 63) / 64));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = stream;
  cfg.numAttrs = 0;
  if (cudaLaunchKernelEx(&cfg, kern, a, gmap, xmap) != cudaSuccess) return FAIRY2I_ERR_CUDA;
  return FAIRY2I_OK;
}

size_t scale_grad_workspace_bytes() { return (size_t)gr::kRedBlocks * 8 * sizeof(double); }

fairy2i_status launch_scale_grad(const float* U, const float* W, int64_t n, int64_t m, int64_t ldc,
                                 int T, const uint32_t* codes, const float* scales, const float* dU,
                                 const float* dW, int64_t ldg, float* rU, float* rW, int64_t ldr,
                                 float* shat, void* ws, cudaStream_t stream) {
  using namespace gr;
  const int64_t row_tiles = (n + 15) / 16, wpr = (m + 127) / 128 * 8;
  double* part = static_cast<double*>(ws);
  zero_kernel<<<304, 256, 0, stream>>>(rU, n, 2 * m, 2 * ldr);
  zero_kernel<<<304, 256, 0, stream>>>(rW, n, 2 * m, 2 * ldr);
  for (int t = T - 1; t >= 0; --t) {
    scale_reduce_kernel<<<kRedBlocks, kRedThreads, 0, stream>>>(dU, dW, ldg, rU, rW, ldr, codes, n,
                                                                m, row_tiles, wpr, t, part);
    scale_update_kernel<<<kRedBlocks, kRedThreads, 0, stream>>>(U, W, ldc, scales, codes, n, m,
                                                                row_tiles, wpr, t, part,
                                                                kRedBlocks, rU, rW, ldr, shat);
  }
  return launch_status();
}

}  // namespace fairy2i
