// C ABI of the library: argument validation, the per-device status word, dispatch.
#include <cuda_runtime.h>

#include <atomic>
#include <mutex>

#include "common.cuh"

namespace fairy2i {

fairy2i_status launch_convert(const float* R, int64_t rows, int64_t cols, int64_t ldR, int64_t n,
                              int64_t m, float* U, float* W, int64_t ldc, cudaStream_t stream);
size_t quantize_workspace_bytes(int64_t n, int64_t m);
fairy2i_status launch_quantize(const float* U, const float* W, int64_t n, int64_t m, int64_t ldc,
                               int T, uint32_t* codes, float* scales, void* workspace,
                               cudaStream_t stream);
fairy2i_status launch_wl_simple(const void* x, fairy2i_dtype xdt, int64_t B, int64_t in_features,
                                int64_t ldx, const uint32_t* codes, const float* scales,
                                int64_t n, int64_t m, int64_t out_features, int64_t wpr, int T,
                                float* y, int64_t ldy, cudaStream_t stream);
fairy2i_status launch_wl_decode(const void* x, fairy2i_dtype xdt, int64_t B, int64_t in_features,
                                int64_t ldx, const uint32_t* codes, const float* scales,
                                int64_t n, int64_t m, int64_t out_features, int64_t wpr, int T,
                                float* y, int64_t ldy, cudaStream_t stream, bool* handled);
fairy2i_status launch_wl_prefill(const void* x, fairy2i_dtype xdt, int64_t B, int64_t in_features,
                                 int64_t ldx, const uint32_t* codes, const float* scales,
                                 int64_t n, int64_t m, int64_t out_features, int64_t wpr, int T,
                                 float* y, int64_t ldy, cudaStream_t stream, bool* handled);
fairy2i_status launch_wl_prefill_group(const void* x, fairy2i_dtype xdt, int64_t B,
                                       int64_t in_features, int64_t ldx, int count,
                                       const uint32_t* const* codes, const float* const* scales,
                                       int64_t n, int64_t m, int64_t out_features, int64_t wpr,
                                       int T, float* const* y, int64_t ldy, cudaStream_t stream,
                                       bool* handled);
fairy2i_status launch_wl_stream_group(const void* x, fairy2i_dtype xdt, int64_t B,
                                      int64_t in_features, int64_t ldx, int count,
                                      const uint32_t* const* codes, const float* const* scales,
                                      int64_t n, int64_t m, int64_t out_features, int64_t wpr,
                                      int T, float* const* y, int64_t ldy, cudaStream_t stream,
                                      bool* handled);
fairy2i_status launch_selftest_wait(uint32_t limit_us, cudaStream_t stream);
fairy2i_status launch_wl_chain(const fairy2i_chain_call* calls, int ncalls, int T,
                               int cluster_size, unsigned int* done, cudaStream_t stream,
                               int nb = 1, int64_t ldx = 0, int64_t ldy = 0);
int chain_max_calls();
size_t ste_grad_workspace_bytes(int64_t B, int64_t in_features, int64_t out_features);
fairy2i_status launch_ste_grad(const void* x, int64_t ldx, const void* g, int64_t ldg, int64_t B,
                               int64_t in_features, int64_t out_features, float* dU, float* dW,
                               int64_t ldc, int accumulate, void* ws, cudaStream_t stream);
size_t scale_grad_workspace_bytes();
fairy2i_status launch_scale_grad(const float* U, const float* W, int64_t n, int64_t m, int64_t ldc,
                                 int T, const uint32_t* codes, const float* scales, const float* dU,
                                 const float* dW, int64_t ldg, float* rU, float* rW, int64_t ldr,
                                 float* shat, void* ws, cudaStream_t stream);
size_t attention_workspace_bytes(int64_t n, int heads, int64_t L);
fairy2i_status launch_attention(const float* q, const float* kc, const float* vc, int64_t L,
                                int64_t ldkv, int64_t n, int heads, float* out, void* ws,
                                size_t ws_bytes, cudaStream_t stream);
fairy2i_status launch_rmsnorm(const float* h, const float* delta, const float* w, int64_t B,
                              int64_t d, float eps, float* h_out, float* out, cudaStream_t stream);
fairy2i_status launch_silu_mul(const float* g, const float* u, int64_t count, float* out,
                               cudaStream_t stream);
fairy2i_status launch_codes_adjoint(const uint32_t* codes, int64_t n, int64_t m, int T,
                                    uint32_t* codes_adj, cudaStream_t stream);
fairy2i_status launch_wl_decode_group(const void* x, fairy2i_dtype xdt, int64_t B,
                                      int64_t in_features, int64_t ldx, int count,
                                      const uint32_t* const* codes, const float* const* scales,
                                      int64_t n, int64_t m, int64_t out_features, int64_t wpr,
                                      int T, float* const* y, int64_t ldy, cudaStream_t stream,
                                      bool* handled);

// Status word: one __device__ word per device that has loaded the module; its address is
// looked up once per device with that device current.
__device__ unsigned int g_status_word;
static unsigned int* g_status_ptr[64];
static std::mutex g_status_mu;

unsigned int* device_status_word() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(g_status_mu);
  if (!g_status_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) return nullptr;
    g_status_ptr[dev] = static_cast<unsigned int*>(p);
  }
  return g_status_ptr[dev];
}

static bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Largest batch the automatic path sends to the chained kernel first (skinny-batch decode: one
// launch of up to 4 tokens per call); larger batches take the tcgen05 prefill GEMM, and the
// chained kernel up to kChainMaxTokens what the GEMM does not take (float32 x, unaligned rows).
// Measured per 7B layer (bf16, T = 2): the chained kernel 77-84 us at 2-4 tokens and 126-142 us
// at 5-8 (two launches per call), the GEMM with K split ~112 us at 2-16.
constexpr int64_t kSkinnyMaxTokens = 4;
constexpr int64_t kChainMaxTokens = 8;

// The automatic decode path (B <= 2 tokens): one token at a time through a kernel that holds
// every x entry to the per-element bound for any x, i.e. to 2^-26 (persistent tcgen05 kernel,
// one-token form, bf16 x) or 2^-28 (chained kernel, float32 x) of the largest |x| in the K slice
// one CTA handles (at most 3072 and 12288 values). *handled = false (nothing launched) where
// neither kernel takes the shape.
static fairy2i_status auto_decode(const void* x, fairy2i_dtype xdt, int64_t B, int64_t in_features,
                                  int64_t ldx, int count, const uint32_t* const* codes,
                                  const float* const* scales, int64_t n, int64_t m,
                                  int64_t out_features, int64_t wpr, int T, float* const* y,
                                  int64_t ldy, cudaStream_t s, bool* handled) {
  *handled = false;
  const int64_t esz = xdt == FAIRY2I_BF16 ? 2 : 4;
  if (xdt == FAIRY2I_F32) {   // chained kernel: T <= 4, in_features <= 24576, x 16-byte aligned
    if (T > 4 || in_features > 24576 || (B > 1 && (ldx * esz) % 16 != 0)) return FAIRY2I_OK;
  }
  for (int64_t b = 0; b < B; ++b) {
    const void* xb = static_cast<const char*>(x) + b * ldx * esz;
    float* yb[FAIRY2I_MAX_GROUP];
    for (int g = 0; g < count; ++g) yb[g] = y[g] + b * ldy;
    if (xdt == FAIRY2I_BF16) {
      bool h = false;
      const fairy2i_status st = launch_wl_stream_group(xb, xdt, 1, in_features, ldx, count, codes,
                                                       scales, n, m, out_features, wpr, T, yb,
                                                       ldy, s, &h);
      if (st != FAIRY2I_OK) return st;
      if (!h) return FAIRY2I_OK;   // the same shape for every token: only b = 0 gets here
    } else {
      fairy2i_chain_call c = {};
      c.x = xb;
      c.xdt = xdt;
      c.count = count;
      c.in_features = in_features;
      c.out_features = out_features;
      for (int g = 0; g < count; ++g) {
        c.codes[g] = codes[g];
        c.scales[g] = scales[g];
        c.y[g] = yb[g];
      }
      const fairy2i_status st = fairy2i_wl_matmul_chain(&c, 1, T, 0, nullptr, 0, s);
      if (st != FAIRY2I_OK) return st;
    }
  }
  *handled = true;
  return FAIRY2I_OK;
}

// B tokens of one call (a group of `count` linears) through the chained kernel, in launches of
// up to 4 tokens (each a block of consecutive rows of x and y): the skinny-batch decode. The
// decoded signs of every unit feed the MMAs of all tokens of a launch; each x entry is held to
// 2^-28 of the largest |x| of its token in the CTA's K slice, so the per-element bound holds for
// any x. *handled = false (nothing launched) outside the kernel's limits (T <= 4,
// in_features <= 24576, x 16-byte aligned).
static fairy2i_status chain_tokens(const void* x, fairy2i_dtype xdt, int64_t B,
                                   int64_t in_features, int64_t ldx, int count,
                                   const uint32_t* const* codes, const float* const* scales,
                                   int64_t out_features, int T, float* const* y, int64_t ldy,
                                   cudaStream_t s, bool* handled) {
  *handled = false;
  const int64_t esz = xdt == FAIRY2I_BF16 ? 2 : 4;
  if (T > 4 || in_features > 24576 || !aligned(x, 16)) return FAIRY2I_OK;
  for (int64_t b0 = 0; b0 < B;) {
    int nb = (int)(B - b0 >= 4 ? 4 : B - b0);
    fairy2i_chain_call c = {};
    c.x = static_cast<const char*>(x) + b0 * ldx * esz;
    c.xdt = xdt;
    c.count = count;
    c.in_features = in_features;
    c.out_features = out_features;
    for (int g = 0; g < count; ++g) {
      c.codes[g] = codes[g];
      c.scales[g] = scales[g];
      c.y[g] = y[g] + b0 * ldy;
    }
    fairy2i_status st;
    for (;;) {   // fewer tokens per launch where the B tiles of nb do not fit
      st = launch_wl_chain(&c, 1, T, 0, nullptr, s, nb, ldx, ldy);
      if (st != FAIRY2I_ERR_INVALID_ARG || nb == 1) break;
      --nb;
    }
    if (st == FAIRY2I_ERR_INVALID_ARG && b0 == 0) return FAIRY2I_OK;
    if (st != FAIRY2I_OK) return st;
    b0 += nb;
  }
  *handled = true;
  return FAIRY2I_OK;
}

}  // namespace fairy2i

using namespace fairy2i;

extern "C" {

const char* fairy2i_status_string(fairy2i_status s) {
  switch (s) {
    case FAIRY2I_OK: return "ok";
    case FAIRY2I_ERR_INVALID_ARG: return "invalid argument";
    case FAIRY2I_ERR_SHAPE: return "shape or leading dimension error";
    case FAIRY2I_ERR_ALIGNMENT: return "misaligned pointer or leading dimension";
    case FAIRY2I_ERR_DTYPE: return "unknown dtype";
    case FAIRY2I_ERR_WORKSPACE: return "workspace missing or too small";
    case FAIRY2I_ERR_NONFINITE: return "non-finite weight";
    case FAIRY2I_ERR_TIMEOUT: return "bounded wait ran out on the device";
    case FAIRY2I_ERR_CUDA: return "CUDA error";
  }
  return "unknown status";
}

fairy2i_status fairy2i_convert(const float* R, int64_t rows, int64_t cols, int64_t ldR, float* U,
                               float* W, int64_t ldc, void* stream) {
  if (!R || !U || !W || rows < 1 || cols < 1) return FAIRY2I_ERR_INVALID_ARG;
  const int64_t n = (rows + 1) / 2, m = (cols + 1) / 2;
  if (ldR < cols || ldc < m) return FAIRY2I_ERR_SHAPE;
  if (!aligned(R, 4) || !aligned(U, 8) || !aligned(W, 8)) return FAIRY2I_ERR_ALIGNMENT;
  return launch_convert(R, rows, cols, ldR, n, m, U, W, ldc, static_cast<cudaStream_t>(stream));
}

int64_t fairy2i_codes_words_per_row(int64_t m) { return m < 1 ? 0 : ((m + 127) / 128) * 8; }

int64_t fairy2i_codes_words(int64_t n, int64_t m, int T) {
  if (n < 1 || m < 1 || T < 1 || T > FAIRY2I_MAX_STAGES) return 0;
  return (int64_t)T * 2 * ((n + 15) / 16) * 16 * fairy2i_codes_words_per_row(m);
}

size_t fairy2i_quantize_workspace_bytes(int64_t n, int64_t m, int T) {
  if (n < 1 || m < 1 || T < 1 || T > FAIRY2I_MAX_STAGES) return 0;
  return quantize_workspace_bytes(n, m);
}

fairy2i_status fairy2i_quantize(const float* U, const float* W, int64_t n, int64_t m, int64_t ldc,
                                int T, uint32_t* codes, float* scales, void* workspace,
                                size_t workspace_bytes, void* stream) {
  if (!U || !W || !codes || !scales || n < 1 || m < 1 || T < 1 || T > FAIRY2I_MAX_STAGES)
    return FAIRY2I_ERR_INVALID_ARG;
  if (n > (int64_t(1) << 40) / m) return FAIRY2I_ERR_SHAPE;
  if (ldc < m) return FAIRY2I_ERR_SHAPE;
  if (!aligned(U, 8) || !aligned(W, 8) || !aligned(codes, 16) || !aligned(scales, 4))
    return FAIRY2I_ERR_ALIGNMENT;
  if (!workspace || workspace_bytes < quantize_workspace_bytes(n, m)) return FAIRY2I_ERR_WORKSPACE;
  if (!aligned(workspace, 256)) return FAIRY2I_ERR_ALIGNMENT;
  return launch_quantize(U, W, n, m, ldc, T, codes, scales, workspace,
                         static_cast<cudaStream_t>(stream));
}

fairy2i_status fairy2i_wl_matmul_path(const void* x, fairy2i_dtype xdt, int64_t B,
                                      int64_t in_features, int64_t ldx, const uint32_t* codes,
                                      const float* scales, int64_t out_features, int T, float* y,
                                      int64_t ldy, int path, void* stream) {
  if (B < 0 || in_features < 1 || out_features < 1 || T < 1 || T > FAIRY2I_MAX_STAGES ||
      path < 0 || path > 5)
    return FAIRY2I_ERR_INVALID_ARG;
  if (xdt != FAIRY2I_F32 && xdt != FAIRY2I_BF16) return FAIRY2I_ERR_DTYPE;
  if (B == 0) return FAIRY2I_OK;
  if (!x || !codes || !scales || !y) return FAIRY2I_ERR_INVALID_ARG;
  if (ldx < in_features || ldy < out_features) return FAIRY2I_ERR_SHAPE;
  if (!aligned(x, 16) || !aligned(codes, 16) || !aligned(y, 4) || !aligned(scales, 4))
    return FAIRY2I_ERR_ALIGNMENT;
  const int64_t n = (out_features + 1) / 2, m = (in_features + 1) / 2;
  const int64_t wpr = fairy2i_codes_words_per_row(m);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  bool handled = false;
  fairy2i_status st = FAIRY2I_OK;
  if (path == 0 && B >= 2 && B <= kSkinnyMaxTokens) {   // skinny batch: chained kernel
    st = chain_tokens(x, xdt, B, in_features, ldx, 1, &codes, &scales, out_features, T, &y, ldy,
                      s, &handled);
    if (handled || st != FAIRY2I_OK) return st;
  }
  if (path == 3 || (path == 0 && B > 2)) {   // tcgen05 prefill GEMM
    st = launch_wl_prefill(x, xdt, B, in_features, ldx, codes, scales, n, m, out_features, wpr, T,
                           y, ldy, s, &handled);
    if (handled || st != FAIRY2I_OK) return st;
    if (path == 3) return FAIRY2I_ERR_INVALID_ARG;   // outside the prefill kernel's domain
  }
  if (path == 0 && B > kSkinnyMaxTokens && B <= kChainMaxTokens) {   // not the GEMM's: chained
    st = chain_tokens(x, xdt, B, in_features, ldx, 1, &codes, &scales, out_features, T, &y, ldy,
                      s, &handled);
    if (handled || st != FAIRY2I_OK) return st;
  }
  if (path == 4) {   // persistent tcgen05 decode kernel (explicit): B <= 2 bf16 tokens, T <= 4
    st = launch_wl_stream_group(x, xdt, B, in_features, ldx, 1, &codes, &scales, n, m,
                                out_features, wpr, T, &y, ldy, s, &handled);
    if (handled || st != FAIRY2I_OK) return st;
    return FAIRY2I_ERR_INVALID_ARG;   // shape or dtype outside the kernel
  }
  if (path == 2) return FAIRY2I_ERR_INVALID_ARG;   // retired
  if (path == 5) {   // the chained decode kernel on this one call, up to 4 tokens a launch
    st = chain_tokens(x, xdt, B, in_features, ldx, 1, &codes, &scales, out_features, T, &y, ldy,
                      s, &handled);
    if (handled || st != FAIRY2I_OK) return st;
    return FAIRY2I_ERR_INVALID_ARG;
  }
  if (path == 0 && B <= 2) {
    st = auto_decode(x, xdt, B, in_features, ldx, 1, &codes, &scales, n, m, out_features, wpr, T,
                     &y, ldy, s, &handled);
    if (handled || st != FAIRY2I_OK) return st;
  }
  if (path == 1) {   // warp-MMA decode kernel (explicit): e4m3 limbs of x
    st = launch_wl_decode(x, xdt, B, in_features, ldx, codes, scales, n, m, out_features, wpr, T,
                          y, ldy, s, &handled);
    if (handled || st != FAIRY2I_OK) return st;
  }
  return launch_wl_simple(x, xdt, B, in_features, ldx, codes, scales, n, m, out_features, wpr, T,
                          y, ldy, s);
}

fairy2i_status fairy2i_wl_matmul(const void* x, fairy2i_dtype xdt, int64_t B, int64_t in_features,
                                 int64_t ldx, const uint32_t* codes, const float* scales,
                                 int64_t out_features, int T, float* y, int64_t ldy,
                                 void* stream) {
  return fairy2i_wl_matmul_path(x, xdt, B, in_features, ldx, codes, scales, out_features, T, y,
                                ldy, 0, stream);
}

fairy2i_status fairy2i_wl_matmul_group_path(const void* x, fairy2i_dtype xdt, int64_t B,
                                            int64_t in_features, int64_t ldx, int count,
                                            const uint32_t* const* codes,
                                            const float* const* scales, int64_t out_features,
                                            int T, float* const* y, int64_t ldy, int path,
                                            void* stream) {
  if (count < 1 || count > FAIRY2I_MAX_GROUP || !codes || !scales || !y ||
      (path != 0 && path != 1 && path != 3 && path != 4 && path != 5))
    return FAIRY2I_ERR_INVALID_ARG;
  // Every member is validated as a single call would be (B = 0 included) before anything runs.
  for (int g = 0; g < count; ++g) {
    if (B < 0 || in_features < 1 || out_features < 1 || T < 1 || T > FAIRY2I_MAX_STAGES)
      return FAIRY2I_ERR_INVALID_ARG;
    if (xdt != FAIRY2I_F32 && xdt != FAIRY2I_BF16) return FAIRY2I_ERR_DTYPE;
    if (B == 0) return FAIRY2I_OK;
    if (!x || !codes[g] || !scales[g] || !y[g]) return FAIRY2I_ERR_INVALID_ARG;
    if (ldx < in_features || ldy < out_features) return FAIRY2I_ERR_SHAPE;
    if (!aligned(x, 16) || !aligned(codes[g], 16) || !aligned(y[g], 4) || !aligned(scales[g], 4))
      return FAIRY2I_ERR_ALIGNMENT;
  }
  const int64_t n = (out_features + 1) / 2, m = (in_features + 1) / 2;
  const int64_t wpr = fairy2i_codes_words_per_row(m);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  bool handled = false;
  if (path == 5 || (path == 0 && B >= 2 && B <= kSkinnyMaxTokens)) {
    // the chained decode kernel on this one group, up to 4 tokens a launch
    const fairy2i_status st = chain_tokens(x, xdt, B, in_features, ldx, count, codes, scales,
                                           out_features, T, y, ldy, s, &handled);
    if (handled || st != FAIRY2I_OK) return st;
    if (path == 5) return FAIRY2I_ERR_INVALID_ARG;
  }
  if (path == 3 || (B > kSkinnyMaxTokens && path == 0)) {   // one prefill GEMM launch
    const fairy2i_status st = launch_wl_prefill_group(x, xdt, B, in_features, ldx, count, codes,
                                                      scales, n, m, out_features, wpr, T, y, ldy,
                                                      s, &handled);
    if (handled || st != FAIRY2I_OK) return st;
    if (path == 3) return FAIRY2I_ERR_INVALID_ARG;   // outside the prefill kernel's domain
  }
  if (path == 0 && B > kSkinnyMaxTokens && B <= kChainMaxTokens) {   // not the GEMM's: chained
    const fairy2i_status st = chain_tokens(x, xdt, B, in_features, ldx, count, codes, scales,
                                           out_features, T, y, ldy, s, &handled);
    if (handled || st != FAIRY2I_OK) return st;
  }
  if (B <= 2 && path == 0) {   // per token, one launch for the whole group
    const fairy2i_status st = auto_decode(x, xdt, B, in_features, ldx, count, codes, scales, n, m,
                                          out_features, wpr, T, y, ldy, s, &handled);
    if (handled || st != FAIRY2I_OK) return st;
  }
  if (B <= 2 && path == 4) {   // one launch of the persistent tcgen05 decode kernel
    const fairy2i_status st = launch_wl_stream_group(x, xdt, B, in_features, ldx, count, codes,
                                                     scales, n, m, out_features, wpr, T, y, ldy,
                                                     s, &handled);
    if (handled || st != FAIRY2I_OK) return st;
    return FAIRY2I_ERR_INVALID_ARG;
  }
  if (B <= 2 && path == 1) {   // one launch of the warp-MMA decode kernel for the whole group
    const fairy2i_status st = launch_wl_decode_group(x, xdt, B, in_features, ldx, count, codes,
                                                     scales, n, m, out_features, wpr, T, y, ldy,
                                                     s, &handled);
    if (handled || st != FAIRY2I_OK) return st;
  }
  for (int g = 0; g < count; ++g) {   // elsewhere: per member
    const fairy2i_status st = fairy2i_wl_matmul_path(x, xdt, B, in_features, ldx, codes[g],
                                                     scales[g], out_features, T, y[g], ldy,
                                                     path == 1 ? 1 : 0, stream);
    if (st != FAIRY2I_OK) return st;
  }
  return FAIRY2I_OK;
}

fairy2i_status fairy2i_wl_matmul_group(const void* x, fairy2i_dtype xdt, int64_t B,
                                       int64_t in_features, int64_t ldx, int count,
                                       const uint32_t* const* codes, const float* const* scales,
                                       int64_t out_features, int T, float* const* y, int64_t ldy,
                                       void* stream) {
  return fairy2i_wl_matmul_group_path(x, xdt, B, in_features, ldx, count, codes, scales,
                                      out_features, T, y, ldy, 0, stream);
}

int fairy2i_wl_matmul_chain_max_calls(void) { return chain_max_calls(); }

size_t fairy2i_wl_matmul_chain_workspace_bytes(int ncalls) {
  if (ncalls <= 1) return 0;
  const int per = chain_max_calls();
  const int counters = ncalls < per ? ncalls : per;
  return ((size_t)counters * sizeof(unsigned int) + 255) & ~(size_t)255;
}

fairy2i_status fairy2i_wl_matmul_chain(const fairy2i_chain_call* calls, int ncalls, int T,
                                       int cluster_size, void* workspace, size_t workspace_bytes,
                                       void* stream) {
  if (!calls || ncalls < 1 || T < 1 || T > 4) return FAIRY2I_ERR_INVALID_ARG;
  if (cluster_size != 0 && cluster_size != 1 && cluster_size != 2 && cluster_size != 4 &&
      cluster_size != 8)
    return FAIRY2I_ERR_INVALID_ARG;
  // Every call is validated before anything is enqueued.
  for (int c = 0; c < ncalls; ++c) {
    const fairy2i_chain_call& k = calls[c];
    if (k.count < 1 || k.count > FAIRY2I_MAX_GROUP || k.in_features < 1 || k.out_features < 1 ||
        !k.x)
      return FAIRY2I_ERR_INVALID_ARG;
    if (k.xdt != FAIRY2I_F32 && k.xdt != FAIRY2I_BF16) return FAIRY2I_ERR_DTYPE;
    if (k.in_features > 24576 || k.out_features > (int64_t(1) << 30))
      return FAIRY2I_ERR_INVALID_ARG;
    if (!aligned(k.x, 16)) return FAIRY2I_ERR_ALIGNMENT;
    for (int g = 0; g < k.count; ++g) {
      if (!k.codes[g] || !k.scales[g] || !k.y[g]) return FAIRY2I_ERR_INVALID_ARG;
      if (!aligned(k.codes[g], 16) || !aligned(k.scales[g], 4) || !aligned(k.y[g], 4))
        return FAIRY2I_ERR_ALIGNMENT;
    }
  }
  const size_t need = fairy2i_wl_matmul_chain_workspace_bytes(ncalls);
  if (need > 0 && (!workspace || workspace_bytes < need)) return FAIRY2I_ERR_WORKSPACE;
  if (need > 0 && !aligned(workspace, 16)) return FAIRY2I_ERR_ALIGNMENT;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int per = chain_max_calls();
  for (int c0 = 0; c0 < ncalls; c0 += per) {
    const int nc = ncalls - c0 < per ? ncalls - c0 : per;
    unsigned int* done = nullptr;
    if (nc > 1) {
      done = static_cast<unsigned int*>(workspace);
      if (cudaMemsetAsync(done, 0, (size_t)nc * sizeof(unsigned int), s) != cudaSuccess)
        return FAIRY2I_ERR_CUDA;
    }
    const fairy2i_status st = launch_wl_chain(calls + c0, nc, T, cluster_size, done, s);
    if (st != FAIRY2I_OK) return st;
  }
  return FAIRY2I_OK;
}

size_t fairy2i_hermitian_attention_workspace_bytes(int64_t n, int heads, int64_t L) {
  return attention_workspace_bytes(n, heads, L);
}

fairy2i_status fairy2i_hermitian_attention(const float* q, const float* k_cache,
                                           const float* v_cache, int64_t L, int64_t ldkv,
                                           int64_t n, int heads, float* out, void* workspace,
                                           size_t workspace_bytes, void* stream) {
  if (!q || !k_cache || !v_cache || !out || L < 1 || n < 1 || heads < 1 || n % heads != 0 ||
      n / heads > 128)
    return FAIRY2I_ERR_INVALID_ARG;
  if (ldkv < 2 * n) return FAIRY2I_ERR_SHAPE;
  if (!aligned(q, 4) || !aligned(k_cache, 4) || !aligned(v_cache, 4) || !aligned(out, 4))
    return FAIRY2I_ERR_ALIGNMENT;
  if (!workspace || workspace_bytes < attention_workspace_bytes(n, heads, L))
    return FAIRY2I_ERR_WORKSPACE;
  if (!aligned(workspace, 4)) return FAIRY2I_ERR_ALIGNMENT;
  return launch_attention(q, k_cache, v_cache, L, ldkv, n, heads, out, workspace, workspace_bytes,
                          static_cast<cudaStream_t>(stream));
}

fairy2i_status fairy2i_rmsnorm(const float* h, const float* delta, const float* w, int64_t B,
                               int64_t d, float eps, float* h_out, float* out, void* stream) {
  if (!h || !w || !out || B < 1 || d < 1 || !(eps >= 0.f) || B > (int64_t(1) << 31))
    return FAIRY2I_ERR_INVALID_ARG;
  if (!aligned(h, 4) || !aligned(w, 4) || !aligned(out, 4) || (delta && !aligned(delta, 4)) ||
      (h_out && !aligned(h_out, 4)))
    return FAIRY2I_ERR_ALIGNMENT;
  return launch_rmsnorm(h, delta, w, B, d, eps, h_out, out, static_cast<cudaStream_t>(stream));
}

fairy2i_status fairy2i_silu_mul(const float* g, const float* u, int64_t count, float* out,
                                void* stream) {
  if (!g || !u || !out || count < 1) return FAIRY2I_ERR_INVALID_ARG;
  if (!aligned(g, 4) || !aligned(u, 4) || !aligned(out, 4)) return FAIRY2I_ERR_ALIGNMENT;
  return launch_silu_mul(g, u, count, out, static_cast<cudaStream_t>(stream));
}

size_t fairy2i_ste_weight_grad_workspace_bytes(int64_t B, int64_t in_features,
                                               int64_t out_features) {
  if (B < 1 || in_features < 1 || out_features < 1) return 0;
  return ste_grad_workspace_bytes(B, in_features, out_features);
}

fairy2i_status fairy2i_ste_weight_grad(const void* x, int64_t ldx, const void* g, int64_t ldg,
                                       int64_t B, int64_t in_features, int64_t out_features,
                                       float* dU, float* dW, int64_t ldc, int accumulate,
                                       void* workspace, size_t workspace_bytes, void* stream) {
  if (!x || !g || !dU || !dW || B < 1 || in_features < 1 || out_features < 1 ||
      B > (int64_t(1) << 26) || in_features > (int64_t(1) << 26) ||
      out_features > (int64_t(1) << 26))
    return FAIRY2I_ERR_INVALID_ARG;
  const int64_t m = (in_features + 1) / 2;
  if (ldx < in_features || ldg < out_features || ldc < m) return FAIRY2I_ERR_SHAPE;
  if (!aligned(x, 2) || !aligned(g, 2) || !aligned(dU, 8) || !aligned(dW, 8))
    return FAIRY2I_ERR_ALIGNMENT;
  if (!workspace || workspace_bytes < ste_grad_workspace_bytes(B, in_features, out_features))
    return FAIRY2I_ERR_WORKSPACE;
  if (!aligned(workspace, 256)) return FAIRY2I_ERR_ALIGNMENT;
  return launch_ste_grad(x, ldx, g, ldg, B, in_features, out_features, dU, dW, ldc, accumulate,
                         workspace, static_cast<cudaStream_t>(stream));
}

size_t fairy2i_scale_grad_workspace_bytes(void) { return scale_grad_workspace_bytes(); }

fairy2i_status fairy2i_scale_grad(const float* U, const float* W, int64_t n, int64_t m,
                                  int64_t ldc, int T, const uint32_t* codes, const float* scales,
                                  const float* dU, const float* dW, int64_t ldg, float* gU,
                                  float* gW, int64_t ldr, float* shat, void* workspace,
                                  size_t workspace_bytes, void* stream) {
  if (!U || !W || !codes || !scales || !dU || !dW || !gU || !gW || !shat || n < 1 || m < 1 ||
      T < 1 || T > FAIRY2I_MAX_STAGES)
    return FAIRY2I_ERR_INVALID_ARG;
  if (n > (int64_t(1) << 40) / m) return FAIRY2I_ERR_SHAPE;
  if (ldc < m || ldg < m || ldr < m) return FAIRY2I_ERR_SHAPE;
  if (!aligned(U, 8) || !aligned(W, 8) || !aligned(dU, 8) || !aligned(dW, 8) || !aligned(gU, 8) ||
      !aligned(gW, 8) || !aligned(codes, 16) || !aligned(scales, 4) || !aligned(shat, 4))
    return FAIRY2I_ERR_ALIGNMENT;
  if (!workspace || workspace_bytes < scale_grad_workspace_bytes()) return FAIRY2I_ERR_WORKSPACE;
  if (!aligned(workspace, 8)) return FAIRY2I_ERR_ALIGNMENT;
  return launch_scale_grad(U, W, n, m, ldc, T, codes, scales, dU, dW, ldg, gU, gW, ldr, shat,
                           workspace, static_cast<cudaStream_t>(stream));
}

fairy2i_status fairy2i_codes_adjoint(const uint32_t* codes, int64_t n, int64_t m, int T,
                                     uint32_t* codes_adj, void* stream) {
  if (!codes || !codes_adj || n < 1 || m < 1 || T < 1 || T > FAIRY2I_MAX_STAGES)
    return FAIRY2I_ERR_INVALID_ARG;
  if (n > (int64_t(1) << 40) / m) return FAIRY2I_ERR_SHAPE;
  if (!aligned(codes, 16) || !aligned(codes_adj, 16)) return FAIRY2I_ERR_ALIGNMENT;
  const uintptr_t a0 = reinterpret_cast<uintptr_t>(codes), b0 = reinterpret_cast<uintptr_t>(codes_adj);
  const uintptr_t a1 = a0 + 4 * (uintptr_t)fairy2i_codes_words(n, m, T);
  const uintptr_t b1 = b0 + 4 * (uintptr_t)fairy2i_codes_words(m, n, T);
  if (a0 < b1 && b0 < a1) return FAIRY2I_ERR_INVALID_ARG;   // the buffers must not overlap
  return launch_codes_adjoint(codes, n, m, T, codes_adj, static_cast<cudaStream_t>(stream));
}

fairy2i_status fairy2i_selftest_wait_timeout(uint32_t limit_us, void* stream) {
  if (limit_us < 1 || limit_us > 100000) return FAIRY2I_ERR_INVALID_ARG;
  return launch_selftest_wait(limit_us, static_cast<cudaStream_t>(stream));
}

fairy2i_status fairy2i_get_status(void* stream) {
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess)
    return FAIRY2I_ERR_CUDA;
  unsigned int* p = device_status_word();
  if (!p) return FAIRY2I_ERR_CUDA;
  unsigned int v = 0;
  if (cudaMemcpy(&v, p, sizeof(v), cudaMemcpyDeviceToHost) != cudaSuccess) return FAIRY2I_ERR_CUDA;
  if (v) {
    const unsigned int zero = 0;
    if (cudaMemcpy(p, &zero, sizeof(zero), cudaMemcpyHostToDevice) != cudaSuccess)
      return FAIRY2I_ERR_CUDA;
  }
  if (v & kStatusTimeout) return FAIRY2I_ERR_TIMEOUT;
  if (v & kStatusNonfinite) return FAIRY2I_ERR_NONFINITE;
  return FAIRY2I_OK;
}

}  // extern "C"
