/*
 * fairy2i.h -- C ABI of the GB300 (sm_103a) Fairy2i widely-linear {+-1, +-i} layer library.
 *
 * The library computes the quantized widely-linear layer of Fairy2i (arXiv 2512.02901):
 *   (1) fairy2i_convert    real map R (2n x 2m)  ->  complex pair U, W     (Sec. 3.1, Eq. UW-from-R)
 *   (2) fairy2i_quantize   U, W -> T stages of 2-bit codes in {+-1, +-i} + per-tensor scales
 *                          (Sec. 3.2 Eq. ifairy-proj / ifairy-scale, Sec. 3.3 residual stages,
 *                           Sec. 3.4 2-bit storage)
 *   (3) fairy2i_wl_matmul  y = sum_t (U^(t) x + W^(t) conj(x)), real layout in and out
 *                          (Eq. widely-linear, Eq. res-sum, Algorithm 1)
 *
 * Conventions shared by every call
 *  - Every pointer is a DEVICE pointer owned by the caller; the library keeps no pointer after
 *    a call returns and allocates no device memory.
 *  - `stream` is a cudaStream_t passed as void* (NULL = the legacy default stream). Calls only
 *    enqueue work on it and never synchronize, except fairy2i_get_status.
 *  - Argument errors are detected on the host before anything is enqueued and returned
 *    synchronously; nothing is written in that case. A failed kernel launch returns
 *    FAIRY2I_ERR_CUDA. Conditions found on the device (a non-finite weight, a bounded wait
 *    that ran out) are latched in a per-device status word read by fairy2i_get_status.
 *  - Real vectors pair their components by halves (Sec. 3.1): x~ = [Re x ; Im x]. A real
 *    dimension that is odd is padded with one zero channel at its end (Sec. 3.1, Remarks) and
 *    the padded output channel is discarded.
 *  - Complex matrices are interleaved (re, im) float32 pairs (the layout of complex64).
 */
#ifndef FAIRY2I_H
#define FAIRY2I_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  FAIRY2I_OK = 0,
  FAIRY2I_ERR_INVALID_ARG = 1, /* null pointer, negative size, T out of range, bad path */
  FAIRY2I_ERR_SHAPE = 2,       /* leading dimension smaller than the row, size mismatch */
  FAIRY2I_ERR_ALIGNMENT = 3,   /* pointer or leading dimension breaks a stated alignment */
  FAIRY2I_ERR_DTYPE = 4,       /* unknown activation dtype */
  FAIRY2I_ERR_WORKSPACE = 5,   /* workspace missing or smaller than the size query */
  FAIRY2I_ERR_NONFINITE = 6,   /* device: a weight given to fairy2i_quantize was inf or NaN */
  FAIRY2I_ERR_TIMEOUT = 7,     /* device: a bounded wait inside a kernel ran out */
  FAIRY2I_ERR_CUDA = 8         /* a CUDA runtime call or kernel launch failed */
} fairy2i_status;

typedef enum { FAIRY2I_F32 = 0, FAIRY2I_BF16 = 1 } fairy2i_dtype;

/* Largest number of residual stages T accepted by every call. */
#define FAIRY2I_MAX_STAGES 8

/* Human-readable name of a status code (static string). */
const char* fairy2i_status_string(fairy2i_status s);

/* ------------------------------------------------------------------------------------------
 * (1) Widely-linear conversion, Sec. 3.1 Eq. UW-from-R (proof of Theorem 1: R = R_lin(U) +
 *     R_conj(W)).
 *   R    float32 [rows][ldR], row-major (an nn.Linear weight: out_features x in_features).
 *   n = ceil(rows/2), m = ceil(cols/2); R is read as a 2n x 2m matrix whose missing last row
 *   and/or column are zero, split into n x m blocks R11 R12 / R21 R22.
 *   U, W complex64 [n][ldc] (ldc counted in complex elements, ldc >= m):
 *     Re U = (R11+R22)/2, Im U = (R21-R12)/2, Re W = (R11-R22)/2, Im W = (R12+R21)/2,
 *   each computed as one float32 add/sub followed by one float32 multiply by 0.5 (IEEE
 *   round-to-nearest-even, no contraction). Columns m..ldc-1 of U, W are not written.
 *   Requirements: rows, cols >= 1; ldR >= cols; ldc >= m; R, U, W 4-byte aligned (U, W 8).
 * ------------------------------------------------------------------------------------------ */
fairy2i_status fairy2i_convert(const float* R, int64_t rows, int64_t cols, int64_t ldR,
                               float* U, float* W, int64_t ldc, void* stream);

/* ------------------------------------------------------------------------------------------
 * (2) PhaseQuant + recursive residual quantization + 2-bit packing (Sec. 3.2-3.4).
 *   For M in {U, W} independently: R^(0) = M; for t = 0..T-1
 *     code c = argmax_{s in {+-1,+-i}} Re(r conj(s)) per element (Eq. ifairy-proj), ties
 *       broken as k = floor(2 Arg(r)/pi + 1/2) breaks them, r = 0 -> +1; codeword i^c;
 *     s_re = mean |Re r| over codes {+-1}, s_im = mean |Im r| over codes {+-i}, per tensor
 *       (Eq. ifairy-scale); an empty set gives 0. Sums are float64 over the row-major element
 *       order in a fixed tree (groups of 256 reduced by v[i] += v[i+h], h = 128..1, the group
 *       sums reduced the same way until one value is left); s = float(S / N);
 *     R^(t+1) = R^(t) - (s_re b_re + i s_im b_im) in float32, one rounding per element
 *       (Sec. 3.3, dequantization and residual update).
 *   U, W     complex64 [n][ldc], read only.
 *   codes    fairy2i_codes_words(n, m, T) uint32 words. Each row of codes is padded with zero
 *            codes to wpr = fairy2i_codes_words_per_row(m) words (16 codes per word, rows
 *            padded to 128 codes) and the rows to 16 R (R = ceil(n/16)) with zero rows; the
 *            buffer is uint32 [T][2][R][wpr/8][16 rows][8 words] (index 1: 0 = U, 1 = W), i.e.
 *            every block of 16 rows x 128 codes is 512 contiguous bytes.
 *            Code k of a row sits in word k/16 at lane i = k%16 as two bits, at
 *            b(i) = 8 (i%2) + i/2 (even codes fill byte 0, odd codes byte 1, in order):
 *              bit b(i)    = 1 iff the codeword has Re+Im < 0  (c in {-1, -i})
 *              bit 16+b(i) = 1 iff the codeword has Re-Im < 0  (c in {+i, -1})
 *            so +1 = (0,0), +i = (0,1), -1 = (1,1), -i = (1,0). Padding is code +1 (0 bits).
 *            T bits per real parameter of R (Sec. 3.4) plus the padding.
 *   scales   float32 [T][2][2]: (s_re, s_im) per (stage, matrix).
 *   workspace >= fairy2i_quantize_workspace_bytes(n, m, T) bytes of device memory, 256-byte
 *            aligned; its contents on entry do not matter and are clobbered.
 *   Requirements: n, m >= 1, n*m < 2^40, 1 <= T <= FAIRY2I_MAX_STAGES, ldc >= m, codes 16-byte
 *   aligned, U, W 8-byte aligned.
 *   A non-finite input element latches FAIRY2I_ERR_NONFINITE (the codes are then unspecified).
 * ------------------------------------------------------------------------------------------ */
int64_t fairy2i_codes_words_per_row(int64_t m);
int64_t fairy2i_codes_words(int64_t n, int64_t m, int T);
size_t fairy2i_quantize_workspace_bytes(int64_t n, int64_t m, int T);
fairy2i_status fairy2i_quantize(const float* U, const float* W, int64_t n, int64_t m,
                                int64_t ldc, int T, uint32_t* codes, float* scales,
                                void* workspace, size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------------------------
 * fairy2i_quantize without a workspace argument. The paper has no counterpart: this is a
 * convenience for callers that cannot allocate device memory at the point of the call, such as
 * a plugin inside a host framework that owns every byte of device memory through its own pool
 * (a raw cudaMalloc there may fail, and a cudaFree synchronizes the whole device), or a
 * latency-bound caller that may not put an allocation on its call path.
 *
 * Same arguments and results as fairy2i_quantize, minus the workspace. The scratch lives in a
 * fixed device array of FAIRY2I_NOALLOC_SCRATCH_BYTES (4 MiB) inside the library, which every
 * GPU that loads the library holds until the process exits. The call allocates nothing and
 * calls no allocating routine.
 *  - Sizes: fairy2i_quantize_workspace_bytes(n, m, T) must not exceed the array, i.e.
 *    n*m <= 16,703,232 complex weights per matrix (a 4096 -> 11008 layer, 5504 x 2048, fits);
 *    larger sizes return FAIRY2I_ERR_WORKSPACE and enqueue nothing.
 *  - The first call on a device looks up the array's device address (cudaGetSymbolAddress,
 *    with that device current); make that first call before any stream capture on the device.
 *  - The array's 4 MiB are committed when the library's device code is loaded on a device. With
 *    CUDA's lazy module loading (the default) that happens at the first call that needs it, and
 *    it can then fail with FAIRY2I_ERR_CUDA if a host framework's pool already holds all device
 *    memory: make the first call on each device before the framework reserves its pool (later
 *    calls commit nothing).
 *  - All calls share the one array, on every stream: calls whose kernels overlap on the GPU
 *    (different streams without ordering between them) race and give wrong results. Calls
 *    ordered on one stream are safe; each call writes every scratch entry before reading it
 *    (its completion counters are cleared by the call itself).
 * ------------------------------------------------------------------------------------------ */
#define FAIRY2I_NOALLOC_SCRATCH_BYTES (4u << 20)
fairy2i_status fairy2i_quantize_noalloc(const float* U, const float* W, int64_t n, int64_t m,
                                        int64_t ldc, int T, uint32_t* codes, float* scales,
                                        void* stream);

/* ------------------------------------------------------------------------------------------
 * (3) Quantized widely-linear matmul (Eq. widely-linear with Eq. res-sum; Algorithm 1 with
 *     the scales placed as in Eq. ifairy-dequant and the W conj(x) term included):
 *       y_b = sum_t sum_{M in {U,W}} sum_k w^(t,M)_{jk} z_k,  z = x_b (U) or conj(x_b) (W),
 *       w^ = s_re b_re + i s_im b_im.
 *   x     [B][ldx] of dtype xdt (float32 or bf16): token b has in_features real entries,
 *         Re x = x[0:m], Im x = x[m:in_features] (+ a zero if in_features is odd),
 *         m = ceil(in_features/2).
 *   codes, scales  as written by fairy2i_quantize for (n, m, T), n = ceil(out_features/2).
 *   y     float32 [B][ldy], overwritten: y[0:n] = Re y, y[n:out_features] = Im y.
 *   Accuracy: every kernel accumulates in fp32. The general (fp32 x) and prefill kernels use x
 *   exactly; the decode kernels hold each x entry in fixed point relative to the largest |x| of
 *   its token in the part of the K range one warp or CTA handles: the one-token persistent
 *   kernel to half a unit of 2^-25 of it, the chained kernel to half a unit of 2^-27, the e4m3
 *   kernels (warp-MMA, two-token persistent: explicit paths only) exactly down to ~2^-13 of it
 *   and to ~2^-22 below. Each output is then within 1e-4 |x~|_1 sum_t max(s_re, s_im) (U and W
 *   terms) of the float64 value for any x on every kernel the automatic path runs, and on the
 *   e4m3 kernels unless hundreds of entries of one part lie in (0, ~2^-13) of its maximum.
 *   Non-finite x: y unspecified.
 *   Requirements: B >= 0 (B = 0 is a no-op), in_features, out_features >= 1, 1 <= T <= 8,
 *   ldx >= in_features, ldy >= out_features, codes and x 16-byte aligned, y 4-byte aligned.
 * ------------------------------------------------------------------------------------------ */
fairy2i_status fairy2i_wl_matmul(const void* x, fairy2i_dtype xdt, int64_t B,
                                 int64_t in_features, int64_t ldx, const uint32_t* codes,
                                 const float* scales, int64_t out_features, int T, float* y,
                                 int64_t ldy, void* stream);

/* Same as fairy2i_wl_matmul with the kernel chosen by `path`:
 *   0 = automatic, every decode choice meeting the per-element bound for any x: B = 1 -> the
 *       persistent tcgen05 kernel's one-token form (4) for bf16 x, the chained kernel (5) for
 *       float32 x; 2 <= B <= 4 -> the chained kernel, one launch (skinny batch); (decode
 *       kernels: T <= 4, in_features <= 24576); B > 4 -> the tcgen05 prefill GEMM where it
 *       applies (see 3), else up to B = 8 the chained kernel (4 tokens per launch); otherwise
 *       the general CUDA-core kernel;
 *   1 = the warp-MMA decode kernel (x as two e4m3 limbs, B <= 2) where it applies, otherwise
 *       the general kernel;
 *   2 = retired (an earlier tcgen05 decode kernel); returns FAIRY2I_ERR_INVALID_ARG;
 *   3 = the tcgen05 prefill GEMM (codes expanded into bf16 +-1 tiles in tensor memory, x by TMA,
 *       64 tokens per tile, 32 up to B = 32; launches of few tiles split K over pairs of CTAs;
 *       T = 3 from B = 512 on as a T = 2 and a T = 1 launch, the second adding into y); it takes
 *       bf16 x with 16-byte aligned rows, ldx % 8 == 0, m % 8 == 0 (m = ceil(in_features/2)) and
 *       T <= 4, and returns FAIRY2I_ERR_INVALID_ARG for anything else;
 *   4 = the persistent tcgen05 decode kernel (one CTA per SM looping over row blocks, the codes
 *       streamed through shared memory and decoded into tensor memory, K split over thread-block
 *       clusters of up to 8 CTAs whose partial rows are summed in rank order; one token: e2m1
 *       operands, each x entry held to 2^-26 of the largest |x| in a CTA's part of the K range,
 *       which keeps every output within the per-element bound for any x; two tokens: e4m3
 *       operands, x as two e4m3 limbs); it takes B <= 2 bf16 tokens, T <= 4 and
 *       in_features <= 24576 and returns FAIRY2I_ERR_INVALID_ARG for anything else;
 *   5 = the chained decode kernel (fairy2i_wl_matmul_chain) on this one call, up to 4 tokens
 *       per launch (the decoded signs feed the MMAs of every token of the launch); it takes any
 *       B (float32 or bf16 x), T <= 4 and in_features <= 24576 and returns
 *       FAIRY2I_ERR_INVALID_ARG for anything else.
 * The tensor-core kernels (paths 1, 3, 4, 5, and so the automatic path) read codes (the decode
 * kernels also the scales) before waiting for the previous kernel in the stream (programmatic
 * dependent launch): the codes must not be written by the kernel launched right before the
 * matmul on the same stream unless that kernel is one of this library's convert/quantize/adjoint
 * kernels, which end before any dependent kernel starts.
 * Results agree within the float32-accumulation tolerance whichever path runs; every kernel sums
 * in a fixed order, so a call repeated with the same shapes on the same device gives the same
 * bits. */
fairy2i_status fairy2i_wl_matmul_path(const void* x, fairy2i_dtype xdt, int64_t B,
                                      int64_t in_features, int64_t ldx, const uint32_t* codes,
                                      const float* scales, int64_t out_features, int T,
                                      float* y, int64_t ldy, int path, void* stream);

/* ------------------------------------------------------------------------------------------
 * Codes of the adjoint layer: the input gradient of the quantized layer (the straight-through
 * backward for x of Sec. 3.2/3.3), x~_grad = R^T y~_grad with R^ = sum_t R_lin(U^(t)) +
 * R_conj(W^(t)). By Eq. realify-ops, R_lin(U)^T = R_lin(U^H) and R_conj(W)^T = R_conj(W^T), so
 * the adjoint is the widely-linear layer U' = U^H, W' = W^T (m x n): the code matrices are
 * transposed, the U codes conjugated (+i <-> -i), and the scales are unchanged. Then
 *   fairy2i_wl_matmul(y_grad, dtype, B, out_features, ldg, codes_adj, scales, in_features, T,
 *                     x_grad, ldxg, stream)
 * computes x~_grad for y~_grad [B][out_features] (the padded output channel of an odd
 * out_features carries no gradient, matching the zero padding of the input).
 *   codes      as written by fairy2i_quantize for (n, m, T): fairy2i_codes_words(n, m, T) words.
 *   codes_adj  fairy2i_codes_words(m, n, T) words, written completely (padding codes 0); must
 *              not overlap codes.
 *   Requirements: n, m >= 1, 1 <= T <= 8, both buffers 16-byte aligned.
 * ------------------------------------------------------------------------------------------ */
fairy2i_status fairy2i_codes_adjoint(const uint32_t* codes, int64_t n, int64_t m, int T,
                                     uint32_t* codes_adj, void* stream);

/* ------------------------------------------------------------------------------------------
 * Several linears of the same shape applied to the same input, e.g. the q, k, v projections
 * or the gate and up projections of a decoder layer: for g < count,
 *   y[g] = fairy2i_wl_matmul(x, xdt, B, in_features, ldx, codes[g], scales[g], out_features, T)
 * with codes[g], scales[g], y[g] device pointers passed in host arrays of `count` entries
 * (1 <= count <= FAIRY2I_MAX_GROUP). Where the automatic decode path applies (B <= 4, T <= 4,
 * in_features <= 24576) the whole group is one launch (B = 1: the persistent tcgen05 kernel's
 * one-token form for bf16 x, the chained kernel for float32 x; 2 <= B <= 4: the chained
 * kernel); B > 4 bf16 tokens on the prefill GEMM: one launch holding every member's tiles (up to
 * B = 8 the chained kernel takes what the GEMM does not, 4 tokens per launch);
 * otherwise the members run one after the other on the automatic path. Requirements and errors are those of fairy2i_wl_matmul
 * for every member (checked before anything is enqueued); FAIRY2I_ERR_INVALID_ARG for a count
 * out of range or a null array. Results agree with the separate calls within the
 * float32-accumulation tolerance (a group splits its work over the SMs differently).
 * ------------------------------------------------------------------------------------------ */
#define FAIRY2I_MAX_GROUP 4
fairy2i_status fairy2i_wl_matmul_group(const void* x, fairy2i_dtype xdt, int64_t B,
                                       int64_t in_features, int64_t ldx, int count,
                                       const uint32_t* const* codes, const float* const* scales,
                                       int64_t out_features, int T, float* const* y, int64_t ldy,
                                       void* stream);

/* fairy2i_wl_matmul_group with the decode kernel chosen by `path`: 0 = automatic (as above),
 * 1 = the warp-MMA decode kernel where it applies (else path 1 per member),
 * 3 = the tcgen05 prefill GEMM, one launch for the group at any B (bf16 x with 16-byte aligned
 * rows, m % 8 == 0, T <= 4; FAIRY2I_ERR_INVALID_ARG otherwise),
 * 4 = the persistent tcgen05 decode kernel, one launch for the group (B <= 2 bf16 tokens, T <= 4,
 * in_features <= 24576; FAIRY2I_ERR_INVALID_ARG for anything else), 5 = the chained decode kernel
 * on this one group (any B, up to 4 tokens per launch, T <= 4, in_features <= 24576;
 * FAIRY2I_ERR_INVALID_ARG otherwise).
 * Any other path returns
 * FAIRY2I_ERR_INVALID_ARG. Results agree with the separate calls within the float32-accumulation
 * tolerance (bit-identical for path 1). */
fairy2i_status fairy2i_wl_matmul_group_path(const void* x, fairy2i_dtype xdt, int64_t B,
                                            int64_t in_features, int64_t ldx, int count,
                                            const uint32_t* const* codes,
                                            const float* const* scales, int64_t out_features,
                                            int T, float* const* y, int64_t ldy, int path,
                                            void* stream);

/* ------------------------------------------------------------------------------------------
 * A chain of one-token calls in one launch: the linears of a decoder applied in data-flow
 * order, e.g. per decoder layer q/k/v (one call of three linears on one input), o, gate/up, down
 * (Eq. widely-linear with Eq. res-sum for every linear; Algorithm 1 with the scales of Eq.
 * ifairy-dequant and the W conj(x) term).
 *   Call c computes, for g < count, y[g] = fairy2i_wl_matmul(x, xdt, 1, in_features,
 *   in_features, codes[g], scales[g], out_features, T, y[g], out_features), and reads x only
 *   after every y of call c - 1 has been written: x of call c may be (a view of) a y of call
 *   c - 1 when xdt is FAIRY2I_F32. The packed codes do not depend on the data and are streamed
 *   ahead across calls.
 *   calls        host array of ncalls descriptors (read before the call returns), 1 <= ncalls.
 *                Chains longer than fairy2i_wl_matmul_chain_max_calls() run as several
 *                launches, one after the other on `stream`.
 *     x          one token: in_features entries of dtype xdt, [Re x | Im x], 16-byte aligned.
 *     codes, scales  as written by fairy2i_quantize for (n, m, T) of that call's shape.
 *     y          out_features float32 values [Re y | Im y] per linear, 4-byte aligned,
 *                overwritten. The y of a call must not overlap its own x or codes, nor another
 *                call's x, y or codes except as the x of the next call.
 *   T            stages, the same for every call, 1 <= T <= 4.
 *   cluster_size 0 picks the K split of the launch; 1, 2, 4 or 8 forces it (thread-block
 *                clusters of that many CTAs split every row; every call then needs
 *                ceil(in_features / 256) >= cluster_size and at most 24 cluster_size
 *                128-code chunks per row).
 *   workspace    >= fairy2i_wl_matmul_chain_workspace_bytes(ncalls) bytes of device memory,
 *                16-byte aligned (completion counters, zeroed by the call on `stream`); may be
 *                NULL when that size is 0 (one call).
 *   Limits: in_features <= 24576 per call (FAIRY2I_ERR_INVALID_ARG otherwise, nothing enqueued).
 *   Accuracy: x is held in fixed point, each entry to 2^-28 of the largest |x| in the part of
 *   the K range one CTA handles; every output is within 1e-4 |x~|_1 sum_t max(s_re, s_im) (U and
 *   W terms) of the float64 value for any x with in_features <= 24576.
 *   The launch keeps one CTA on each SM it uses and its CTAs wait for one another between calls
 *   (bounded: FAIRY2I_ERR_TIMEOUT in the status word after about a second), so a chain should
 *   not share the device with other work that could hold SMs for that long.
 * ------------------------------------------------------------------------------------------ */
typedef struct {
  const void* x;
  fairy2i_dtype xdt;
  int32_t count;                               /* linears sharing x, 1..FAIRY2I_MAX_GROUP */
  int64_t in_features, out_features;
  const uint32_t* codes[FAIRY2I_MAX_GROUP];
  const float* scales[FAIRY2I_MAX_GROUP];
  float* y[FAIRY2I_MAX_GROUP];
} fairy2i_chain_call;

int fairy2i_wl_matmul_chain_max_calls(void);
size_t fairy2i_wl_matmul_chain_workspace_bytes(int ncalls);
fairy2i_status fairy2i_wl_matmul_chain(const fairy2i_chain_call* calls, int ncalls, int T,
                                       int cluster_size, void* workspace, size_t workspace_bytes,
                                       void* stream);

/* ------------------------------------------------------------------------------------------
 * The rest of a widely-linear decoder layer for one token (Sec. 3.1, self-attention in
 * widely-linear form). Vectors use the real layout of the matmul calls: a complex vector of n
 * channels is 2 n floats [Re | Im].
 *
 * Attention with Hermitian scores (Eq. hermitian-score) of one query over L cached positions:
 *   head h is the complex channels [h dc, (h+1) dc), dc = n / heads, d_k = 2 dc;
 *   S[h, l] = Re(q_h^H k_{l,h}) / sqrt(d_k) (the real dot product of the stacked head vectors),
 *   p = softmax over l per head, o_h = sum_l p[h, l] v_{l,h} (real and imaginary parts of v
 *   weighted alike).
 *   q        float32 [2 n]; k_cache, v_cache float32 [L][ldkv] (2 n used per position: a key or
 *            value as fairy2i_wl_matmul writes it, so a call can write the new position's key
 *            and value straight into the caches); out float32 [2 n] (may not overlap the inputs).
 *   workspace >= fairy2i_hermitian_attention_workspace_bytes(n, heads, L) bytes, 4-byte aligned
 *            (per-split partial softmax sums; contents on entry do not matter).
 *   Requirements: L >= 1, heads >= 1, n % heads == 0, dc <= 128, ldkv >= 2 n, pointers 4-byte
 *   aligned. Scores and value sums are accumulated in two-float (compensated) arithmetic.
 *   A real model's head layout (2 dc consecutive real channels per head) maps onto this one by
 *   permuting the output channels of R_Q, R_K, R_V (and the input channels of R_O) before
 *   conversion so that each head's real channels are the real and imaginary parts of dc complex
 *   channels.
 * ------------------------------------------------------------------------------------------ */
size_t fairy2i_hermitian_attention_workspace_bytes(int64_t n, int heads, int64_t L);
fairy2i_status fairy2i_hermitian_attention(const float* q, const float* k_cache,
                                           const float* v_cache, int64_t L, int64_t ldkv,
                                           int64_t n, int heads, float* out, void* workspace,
                                           size_t workspace_bytes, void* stream);

/* RMS normalisation of B tokens of d real values (the decoder's norm layers stay real): with
 * v = h + delta (delta may be NULL), out = v / sqrt(mean(v^2) + eps) * w, and h_out = v when
 * h_out is not NULL (the residual stream after an add). float32 throughout; out and h_out may
 * alias h. Requirements: B >= 1, d >= 1, eps >= 0, pointers 4-byte aligned. */
fairy2i_status fairy2i_rmsnorm(const float* h, const float* delta, const float* w, int64_t B,
                               int64_t d, float eps, float* h_out, float* out, void* stream);

/* The gated activation of the decoder's MLP, out = silu(g) * u elementwise over `count` float32
 * values (out may alias g or u). */
fairy2i_status fairy2i_silu_mul(const float* g, const float* u, int64_t count, float* out,
                                void* stream);

/* ------------------------------------------------------------------------------------------
 * Host (CPU) matmul by look-up tables (Sec. 3.4, LUT-based optimization for CPU), for the host
 * cores of the machine (no GPU involved; every pointer here is HOST memory).
 * fairy2i_lut_quantize_x: int8 activations of one token, per-token symmetric absmax:
 *   delta = float(max |x~_i| / 127) (float32 division), xq_i = round-half-even(x~_i / delta)
 *   clamped to [-127, 127] (all zero when x~ = 0). x float32 [in_features], xq int8
 *   [in_features]; *scale = delta. FAIRY2I_ERR_INVALID_ARG for a non-finite x.
 * fairy2i_lut_matmul: y = delta sum_t (U^(t) z + W^(t) conj(z)), z the complex int8 token
 *   (Re = xq[0:m], Im = xq[m:in_features], zero-padded), codes and scales as fairy2i_quantize
 *   writes them (packed layout, HOST copies), y float32 [out_features] in the real layout.
 *   Four codes of a packed word form one 8-bit index; per group of four inputs a table of 256
 *   entries holds the exact integer partial sums over the real-axis codes and over the
 *   imaginary-axis codes, one table serving U (z) and W (conj(z)). Sums are exact integers,
 *   then scaled in float64: y equals the float64 widely-linear matmul of delta xq to rounding.
 *   workspace >= fairy2i_lut_workspace_bytes(in_features) bytes of host memory (8-byte
 *   aligned); nthreads host threads (1 .. 1024) split the tables and the rows.
 * ------------------------------------------------------------------------------------------ */
fairy2i_status fairy2i_lut_quantize_x(const float* x, int64_t in_features, int8_t* xq,
                                      float* scale);
size_t fairy2i_lut_workspace_bytes(int64_t in_features);
fairy2i_status fairy2i_lut_matmul(const int8_t* xq, float x_scale, int64_t in_features,
                                  const uint32_t* codes, const float* scales,
                                  int64_t out_features, int T, float* y, void* workspace,
                                  size_t workspace_bytes, int nthreads);

/* ------------------------------------------------------------------------------------------
 * Gradients for quantization-aware training (Sec. 3.2 QAT paragraph, Sec. 3.3 QAT).
 *
 * fairy2i_ste_weight_grad: the gradient of a loss with respect to the dequantized pair (U^, W^)
 *   of a layer, which the straight-through estimator passes to the full-precision masters:
 *   dU = sum_b g_b conj(x_b)^T, dW = sum_b g_b x_b^T (complex), from y = U^ x + W^ conj(x).
 *   x   bf16 [B][ldx] real layout (in_features used), the layer input;
 *   g   bf16 [B][ldg] real layout (out_features used), dL/dy~;
 *   dU, dW complex64 [n][ldc] (n = ceil(out/2), m = ceil(in/2), ldc >= m), written, or added
 *   to when accumulate != 0. One real GEMM G = g~^T x~ on the tensor cores (bf16 x bf16 -> f32)
 *   gives both: dU = (G11 + G22) + i (G21 - G12), dW = (G11 - G22) + i (G12 + G21).
 *   workspace >= fairy2i_ste_weight_grad_workspace_bytes(B, in_features, out_features) bytes,
 *   256-byte aligned (token-contiguous copies of x and g). Requirements: B, in, out >= 1,
 *   x, g 2-byte aligned, dU, dW 8-byte aligned.
 *
 * fairy2i_scale_grad: the part of the master gradient that flows through the per-tensor scales
 *   of Eq. ifairy-scale, codes held fixed. For M in {U, W} with dM = dL/dM^ (e.g. from
 *   fairy2i_ste_weight_grad), backpropagating through r^(t+1) = r^(t) - (s_re b_re + i s_im b_im)
 *   and s_re = mean |Re r^(t)| over the +-1 codes (s_im likewise) gives, from r^_T = 0,
 *     s^_t = <dM - r^_(t+1), b^t> (real parts over the +-1 codes, imaginary over the +-i codes),
 *     r^_t = r^_(t+1) + s^_re,t sign(Re r^(t)) / N_re [+-1 codes] + i s^_im,t sign(Im r^(t)) /
 *            N_im [+-i codes];
 *   gU, gW (complex64 [n][ldr]) receive r^_0, shat (float32 [T][2][2]) the total scale
 *   gradients s^. The full master gradient is dM + r^_0. U, W, codes, scales as fairy2i_quantize
 *   read and wrote them (r^(t) is replayed exactly as the quantizer computed it); sums are
 *   float64 in a fixed order. workspace >= fairy2i_scale_grad_workspace_bytes() bytes, 8-byte
 *   aligned. Requirements: n, m >= 1, 1 <= T <= 8, ldc, ldg, ldr >= m.
 * ------------------------------------------------------------------------------------------ */
size_t fairy2i_ste_weight_grad_workspace_bytes(int64_t B, int64_t in_features,
                                               int64_t out_features);
fairy2i_status fairy2i_ste_weight_grad(const void* x, int64_t ldx, const void* g, int64_t ldg,
                                       int64_t B, int64_t in_features, int64_t out_features,
                                       float* dU, float* dW, int64_t ldc, int accumulate,
                                       void* workspace, size_t workspace_bytes, void* stream);
size_t fairy2i_scale_grad_workspace_bytes(void);
fairy2i_status fairy2i_scale_grad(const float* U, const float* W, int64_t n, int64_t m,
                                  int64_t ldc, int T, const uint32_t* codes, const float* scales,
                                  const float* dU, const float* dW, int64_t ldg, float* gU,
                                  float* gW, int64_t ldr, float* shat, void* workspace,
                                  size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------------------------
 * Synchronizes `stream`, then returns and clears the device-side status of the current
 * device: FAIRY2I_ERR_NONFINITE, FAIRY2I_ERR_TIMEOUT, FAIRY2I_ERR_CUDA (an asynchronous CUDA
 * error) or FAIRY2I_OK.
 * ------------------------------------------------------------------------------------------ */
fairy2i_status fairy2i_get_status(void* stream);

/* ------------------------------------------------------------------------------------------
 * Self-test of the device-side failure detection. Enqueues on `stream` one small kernel that
 * runs the bounded barrier wait of the matmul kernels' pipelines on a barrier that nothing
 * completes. After about limit_us microseconds the wait gives up, latches FAIRY2I_ERR_TIMEOUT
 * in the status word (read and cleared by fairy2i_get_status) and the kernel returns normally,
 * so the CUDA context stays usable. limit_us must be in 1 .. 100000
 * (FAIRY2I_ERR_INVALID_ARG otherwise, nothing enqueued); FAIRY2I_ERR_CUDA if the launch fails.
 * ------------------------------------------------------------------------------------------ */
fairy2i_status fairy2i_selftest_wait_timeout(uint32_t limit_us, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* FAIRY2I_H */
