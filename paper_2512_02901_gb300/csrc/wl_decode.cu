// Decode (GEMV, B <= 2 tokens) kernel of the quantized widely-linear matmul on the warp-level
// fp8 tensor cores, with the packed codes staged by TMA.
//
// Arithmetic (Eq. ifairy-dequant, Algorithm 1 with the W conj(x) term). A code carries the two
// sign bits of its codeword b along the diagonals: sigma = sign(Re b + Im b), tau = sign(Re b -
// Im b), so b = ((sigma + tau) + i (sigma - tau))/2 and, with h = (s_re + i s_im)/2,
//     s_re b_re + i s_im b_im = h sigma + conj(h) tau.
// Per (stage t, matrix M) the layer needs the +-1 sums P = sum_k sigma_k x_k and
// Q = sum_k tau_k x_k for every output row; then y += h P + conj(h) Q for U, and
// h conj(P) + conj(h) conj(Q) for W (the conj(x) term of Eq. widely-linear).
//
// Tensor-core form: one m16n8k32 e4m3 MMA chain per (t, M) and 16 rows. Row j of A holds, per
// code k, its sigma-plane and tau-plane entries; B holds x_k in a "sigma" column for the first
// and in a "tau" column for the second. x (bf16, 8 significant bits) is split exactly into two
// e4m3 limbs, hi = e4m3(x S) and lo = e4m3(64 (x S - hi)), with S a power of two per warp and
// token, so the 8 columns are (limb, slot, re/im) and products/sums are fp32.
//
// Decoding: a 32-bit code word holds 16 codes; byte 0 carries the sigma bits of the even codes,
// byte 1 of the odd codes, bytes 2-3 the tau bits likewise. Register j (j = 0..7) of A takes
// bit j of every byte -- K elements (sigma_2j, sigma_2j+1, tau_2j, tau_2j+1) -- after a left
// shift by 2 for j in {0,1,4,5}, so that every bit sits at position q in {2, 3, 6, 7} of its
// byte; one LOP3 then turns each byte into an e4m3 value affine in the bit (bit = 1 for a
// negative sign):
//     q = 7:  (w & 0x80) ^ 0xB8  ->  -1 + 2 bit      q = 6:  (w & 0x40)        ->  0 + 2 bit
//     q = 3:  (w & 0x08) | 0x40  ->   2 + 2 bit      q = 2:  (w & 0x04) | 0x48 ->  4 + 2 bit
// i.e. a = alpha_q + 2 bit and sigma = 1 - 2 bit = (1 + alpha_q) - a. Hence P = C - D with D
// the MMA result and C = sum_k (1 + alpha(k)) x_k, one constant per token and K range shared by
// every row, stage and matrix (and by the tau plane).
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_fp8.h>

#include <mutex>

#include "common.cuh"
#include "ptx.cuh"

namespace fairy2i {

namespace dec {

constexpr int kWarps = 16;
constexpr int kThreads = kWarps * 32;
constexpr int kRows = 16;                     // output rows per CTA (one MMA row tile)
constexpr int kChunkWords = 8;                // words per row per chunk (128 codes)
constexpr int kChunkCodes = kChunkWords * 16;
constexpr int kTileWords = kRows * kChunkWords;
constexpr int kTileBytes = kTileWords * 4;    // 512 B per (chunk, stage-matrix)
constexpr int kXBytes = 576;                  // staged e4m3 x of one chunk and token (2 limbs)
constexpr int kMaxChunksPerWarp = 8;
constexpr uint32_t kWaitLimit = 1u << 22;
constexpr int kMaxSmem = 200 * 1024;

constexpr int kMaxGroup = 4;                 // linears of one launch that share x

struct Args {
  const uint32_t* codes[kMaxGroup];      // per linear of the group (same shape, same x)
  const float* scales[kMaxGroup];
  float* y[kMaxGroup];
  const __nv_bfloat16* x;
  int64_t B, in_features, ldx;
  int64_t n, m, out_features, ldy;
  int wpr, nchunks;
  int tiles;             // 16-row tiles per linear: CTA blockIdx.x works on linear
                         // blockIdx.x / tiles, row tile blockIdx.x % tiles
  int x_vec;             // x rows 16-byte aligned with m % 8 == 0: vector loads allowed
  unsigned int* status;
  int x_off, raw_off, red_off, bar_off, cpw;
};

// Constants of the decode, kept in registers so that every A register costs one LOP3.
struct DecodeConsts {
  uint32_t m2, m3, m6, m7, c2, c7;
};

// A register j of a word: K elements (sigma_2j, sigma_2j+1, tau_2j, tau_2j+1) as e4m3, from the
// word w0 and w2 = w0 << 2; the codes 2j, 2j+1 get the weight 1 + alpha = 5, 3, 5, 3, 1, 0, 1, 0
// for j = 0..7 (bit position 2, 3, 2, 3, 6, 7, 6, 7 of each byte).
template <int J>
__device__ __forceinline__ uint32_t decode_reg(uint32_t w0, uint32_t w2, const DecodeConsts& k) {
  constexpr bool shifted = (J == 0 || J == 1 || J == 4 || J == 5);
  constexpr int q = shifted ? J + 2 : J;      // bit position inside each byte
  const uint32_t w = shifted ? w2 : w0;
  if constexpr (q == 7) return lop3_and_xor(w, k.m7, k.c7);      // -1 + 2 bit
  else if constexpr (q == 6) return w & k.m6;                    //  0 + 2 bit
  else if constexpr (q == 3) return lop3_and_or(w, k.m3, k.m6);  //  2 + 2 bit (0x40 = 2.0)
  else return lop3_and_or(w, k.m2, k.c2);                        //  4 + 2 bit
}

__device__ __forceinline__ void mma_e4m3(float d[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k32.row.col.f32.e4m3.e4m3.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ float bf_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

// Eight bf16 x values of one part (re/im) of token `b` starting at complex index k (k % 8 == 0),
// zero outside [0, m) and beyond in_features.
__device__ __forceinline__ uint4 load_x8(const Args& a, int b, int part, int k) {
  const __nv_bfloat16* row = a.x + (int64_t)b * a.ldx + (int64_t)part * a.m;
  const int64_t lim = part ? a.in_features - a.m : a.m;   // valid complex indices of this part
  if (a.x_vec && k + 8 <= lim) return __ldg(reinterpret_cast<const uint4*>(row + k));
  uint32_t w[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int k0 = k + 2 * i, k1 = k0 + 1;
    const uint32_t lo = k0 < lim ? (uint32_t)__bfloat16_as_ushort(row[k0]) : 0u;
    const uint32_t hi = k1 < lim ? (uint32_t)__bfloat16_as_ushort(row[k1]) : 0u;
    w[i] = lo | (hi << 16);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

__device__ __forceinline__ uint32_t e4m3x2(float a, float b) {
  return (uint32_t)__nv_cvt_float2_to_fp8x2(make_float2(a, b), __NV_SATFINITE, __NV_E4M3);
}

// Power-of-two scale S with max|x| S < 128 (and 1/S), from the exponent bits of max|x|.
__device__ __forceinline__ void pow2_scale(float mx, float& S, float& invS) {
  const int E = (int)((__float_as_uint(mx) >> 23) & 0xffu);
  if (E >= 7 && E <= 254) {
    S = __uint_as_float((uint32_t)(260 - E) << 23);
    invS = __uint_as_float((uint32_t)(E - 6) << 23);
  } else {
    S = 1.f;
    invS = 1.f;
  }
}

// e4m3 limbs of two scaled values (|v| < 128): hi = e4m3(v) rounded to nearest, lo =
// e4m3(64 (v - hi)); |v - hi| <= 2^-4 |v| so |lo| < 2^8, and lo carries the remaining bits of a
// bf16 input exactly whenever hi is a normal e4m3 number.
__device__ __forceinline__ void limbs2(float v0, float v1, uint32_t& hi, uint32_t& lo) {
  hi = e4m3x2(v0, v1);
  const float2 h = __half22float2(__half2(__nv_cvt_fp8x2_to_halfraw2((__nv_fp8x2_storage_t)hi, __NV_E4M3)));
  lo = e4m3x2(64.f * (v0 - h.x), 64.f * (v1 - h.y));
}

template <int NB, int T>
__global__ void __launch_bounds__(kThreads, 1) wl_decode_fp8_kernel(const Args a) {
  constexpr int T2 = 2 * T;
  extern __shared__ __align__(1024) unsigned char smem[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int g = lane >> 2, t4 = lane & 3;
  int lin = 0, tile = (int)blockIdx.x;   // linear of the group and row tile (count <= 4)
  while (tile >= a.tiles) {
    tile -= a.tiles;
    ++lin;
  }
  const uint32_t* const codes = a.codes[lin];
  const float* const scales = a.scales[lin];
  // The scales, like the codes, are not written by the previous kernel: read them now, so that
  // their latency is not paid after the MMAs.
  float scl[T2][2];
#pragma unroll
  for (int tm = 0; tm < T2; ++tm) {
    scl[tm][0] = __ldg(scales + tm * 2 + 0);
    scl[tm][1] = __ldg(scales + tm * 2 + 1);
  }
  const int64_t j0 = (int64_t)tile * kRows;
  const uint32_t* codes_s = reinterpret_cast<const uint32_t*>(smem);
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + a.bar_off) + warp;
  unsigned char* xw = smem + a.x_off + (size_t)warp * a.cpw * NB * kXBytes;
  uint4* xraw = reinterpret_cast<uint4*>(smem + a.raw_off) + (size_t)warp * a.cpw * NB * 32;
  float* red = reinterpret_cast<float*>(smem + a.red_off);
  // This warp's chunks: an even split of the nchunks 128-code chunks of every row.
  const int c_begin = (warp * a.nchunks) / kWarps, c_end = ((warp + 1) * a.nchunks) / kWarps;
  const int nc = c_end - c_begin;

  // Prologue (weights only): each warp bulk-copies its contiguous chunk range of every
  // (stage, matrix) block of this row tile (16 rows x 128 codes = 512 B per chunk, the chunks
  // of a row tile adjacent) and owns the barrier; no CTA-wide barrier is needed.
  if (lane == 0) {
    mbar_init(bar, 1);
    fence_mbar_init();
    if (nc > 0) {
      mbar_arrive_expect_tx(bar, (uint32_t)(T2 * nc * kTileBytes));
      const int64_t tiles = (a.n + kRows - 1) / kRows;
#pragma unroll
      const uint64_t pol = l2_evict_first_policy();   // the codes are read once per launch
      for (int tm = 0; tm < T2; ++tm)
        bulk_load_hint(smem + (size_t)(tm * a.nchunks + c_begin) * kTileBytes,
                       codes + ((tm * tiles + tile) * a.nchunks + c_begin) * kTileWords,
                       (uint32_t)(nc * kTileBytes), bar, pol);
    }
  }
  __syncwarp();
  pdl_launch_dependents();
  // Activations may come from the previous kernel in the stream.
  pdl_wait_primary();

  // Stage this warp's K range of x as e4m3 limbs. Lane l covers part l>>4 (re/im) and the 8
  // values at (l&15)*8 of each chunk: positions 8h..8h+7 (h = l&1) of block (l&15)>>1.
  const int xpart = lane >> 4, xk = (lane & 15) * 8, xh = lane & 1;
  float Cw[NB], invS[NB];
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    float mx = 0.f, cacc = 0.f;
    for (int i = 0; i < nc; ++i) {
      const uint4 u = b < a.B ? load_x8(a, b, xpart, (c_begin + i) * kChunkCodes + xk)
                              : make_uint4(0, 0, 0, 0);
      xraw[(i * NB + b) * 32 + lane] = u;       // kept for the second pass
      const uint32_t v[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) mx = fmaxf(mx, fmaxf(fabsf(bf_lo(v[e])), fabsf(bf_hi(v[e]))));
      // 1 + alpha per pair of positions: 5,3,5,3 (first half of a block), 1,0,1,0 (second)
      const float p0 = bf_lo(v[0]) + bf_hi(v[0]), p1 = bf_lo(v[1]) + bf_hi(v[1]);
      const float p2 = bf_lo(v[2]) + bf_hi(v[2]), p3 = bf_lo(v[3]) + bf_hi(v[3]);
      cacc += xh ? (p0 + p2) : (5.f * (p0 + p2) + 3.f * (p1 + p3));
    }
#pragma unroll
    for (int h = 16; h >= 1; h >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, h));
#pragma unroll
    for (int h = 8; h >= 1; h >>= 1) cacc += __shfl_xor_sync(0xffffffffu, cacc, h);
    Cw[b] = cacc;                               // lanes 0-15: re part, 16-31: im part
    float S;
    pow2_scale(mx, S, invS[b]);
    for (int i = 0; i < nc; ++i) {      // second pass: this lane's own staged values
      const uint4 u = xraw[(i * NB + b) * 32 + lane];
      const uint32_t v[4] = {u.x, u.y, u.z, u.w};
      uint32_t hw[2], lw[2];
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        uint32_t h0, l0, h1, l1;
        limbs2(bf_lo(v[2 * e]) * S, bf_hi(v[2 * e]) * S, h0, l0);
        limbs2(bf_lo(v[2 * e + 1]) * S, bf_hi(v[2 * e + 1]) * S, h1, l1);
        hw[e] = h0 | (h1 << 16);
        lw[e] = l0 | (l1 << 16);
      }
      unsigned char* dst =
          xw + (size_t)(i * NB + b) * kXBytes + xpart * 144 + ((lane & 15) >> 1) * 16 + xh * 8;
      *reinterpret_cast<uint2*>(dst) = make_uint2(hw[0], hw[1]);
      *reinterpret_cast<uint2*>(dst + 288) = make_uint2(lw[0], lw[1]);
    }
  }
  __syncwarp();

  // B column g: limb g>>2 (hi, lo), slot (g>>1)&1 (sigma, tau), part g&1 (re, im).
  const int limb = g >> 2, slot = (g >> 1) & 1, part = g & 1;
  float acc[NB][T2][4];
#pragma unroll
  for (int b = 0; b < NB; ++b)
#pragma unroll
    for (int tm = 0; tm < T2; ++tm) acc[b][tm][0] = acc[b][tm][1] = acc[b][tm][2] = acc[b][tm][3] = 0.f;
  const bool ok = nc == 0 || mbar_wait_bounded(bar, 0, kWaitLimit);
  // Shared-memory addresses: this lane's two code words (rows g and g+8) of a (stage-matrix,
  // chunk) tile and its 16-byte B source in the staged x of a chunk.
  const uint32_t sa_codes = smem_u32(smem) + (uint32_t)(c_begin * kTileBytes) + g * 32 + t4 * 8;
  const uint32_t tm_stride = (uint32_t)(a.nchunks * kTileBytes);
  const uint32_t sa_x = smem_u32(xw) + limb * 288 + part * 144 + t4 * 32;
  // B register = two e4m3 pairs (x_a, x_b) placed in the sigma half (bytes 0-1) or tau half.
  const uint32_t sel0 = slot ? 0x1044u : 0x4410u, sel1 = slot ? 0x3244u : 0x4432u;
  const DecodeConsts k{0x04040404u, 0x08080808u, 0x40404040u, 0x80808080u, 0x48484848u,
                       0xB8B8B8B8u};
  for (int i = 0; ok && i < nc; ++i) {
    uint2 wg[T2], wh[T2];
#pragma unroll
    for (int tm = 0; tm < T2; ++tm) {
      wg[tm] = lds64(sa_codes + tm * tm_stride + i * kTileBytes);
      wh[tm] = lds64(sa_codes + tm * tm_stride + i * kTileBytes + 8 * 32);
    }
#pragma unroll
    for (int ww = 0; ww < 2; ++ww) {
      uint32_t b0[NB][4], b1[NB][4];
#pragma unroll
      for (int b = 0; b < NB; ++b) {
        const uint4 xv = lds128(sa_x + (uint32_t)((i * NB + b) * kXBytes) + ww * 16);
        const uint32_t px[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          b0[b][e] = prmt(px[e], 0u, sel0);
          b1[b][e] = prmt(px[e], 0u, sel1);
        }
      }
      // The T2 stage-matrix accumulators are independent: issue their MMAs round-robin.
      uint32_t gw[T2][2], hw[T2][2];
#pragma unroll
      for (int tm = 0; tm < T2; ++tm) {
        gw[tm][0] = ww ? wg[tm].y : wg[tm].x;
        hw[tm][0] = ww ? wh[tm].y : wh[tm].x;
        gw[tm][1] = gw[tm][0] << 2;
        hw[tm][1] = hw[tm][0] << 2;
      }
#pragma unroll
      for (int b = 0; b < NB; ++b) {
#pragma unroll
        for (int tm = 0; tm < T2; ++tm)
          mma_e4m3(acc[b][tm], decode_reg<0>(gw[tm][0], gw[tm][1], k),
                   decode_reg<0>(hw[tm][0], hw[tm][1], k), decode_reg<1>(gw[tm][0], gw[tm][1], k),
                   decode_reg<1>(hw[tm][0], hw[tm][1], k), b0[b][0], b1[b][0]);
#pragma unroll
        for (int tm = 0; tm < T2; ++tm)
          mma_e4m3(acc[b][tm], decode_reg<2>(gw[tm][0], gw[tm][1], k),
                   decode_reg<2>(hw[tm][0], hw[tm][1], k), decode_reg<3>(gw[tm][0], gw[tm][1], k),
                   decode_reg<3>(hw[tm][0], hw[tm][1], k), b0[b][1], b1[b][1]);
#pragma unroll
        for (int tm = 0; tm < T2; ++tm)
          mma_e4m3(acc[b][tm], decode_reg<4>(gw[tm][0], gw[tm][1], k),
                   decode_reg<4>(hw[tm][0], hw[tm][1], k), decode_reg<5>(gw[tm][0], gw[tm][1], k),
                   decode_reg<5>(hw[tm][0], hw[tm][1], k), b0[b][2], b1[b][2]);
#pragma unroll
        for (int tm = 0; tm < T2; ++tm)
          mma_e4m3(acc[b][tm], decode_reg<6>(gw[tm][0], gw[tm][1], k),
                   decode_reg<6>(hw[tm][0], hw[tm][1], k), decode_reg<7>(gw[tm][0], gw[tm][1], k),
                   decode_reg<7>(hw[tm][0], hw[tm][1], k), b0[b][3], b1[b][3]);
      }
    }
  }
  if (!ok) latch_status(a.status, kStatusTimeout);

  // Epilogue. Lane (g, t4) holds columns 2 t4, 2 t4 + 1 of rows g, g+8: t4 = 0 (hi, P_D),
  // 1 (hi, Q_D), 2 (lo, P_D), 3 (lo, Q_D), P = C - P_D, Q = C - Q_D. The D part of
  // y = sum h P + conj(h) Q (conjugated for W) is accumulated per lane, unscaled, and the
  // limbs and slots are added across lanes; the C part, sum_t s_re^U C + s_re^W conj(C),
  // is added once per warp.
  const bool is_q = t4 & 1;
  float sre_u = 0.f, sre_w = 0.f;
#pragma unroll
  for (int t = 0; t < T; ++t) {
    sre_u += scl[t * 2 + 0][0];
    sre_w += scl[t * 2 + 1][0];
  }
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    const float cre = __shfl_sync(0xffffffffu, Cw[b], 0);
    const float cim = __shfl_sync(0xffffffffu, Cw[b], 16);
    float yr0 = 0.f, yi0 = 0.f, yr1 = 0.f, yi1 = 0.f;   // rows g, g+8
#pragma unroll
    for (int tm = 0; tm < T2; ++tm) {
      const int t = tm >> 1, mat = tm & 1;
      const float hr = 0.5f * scl[t * 2 + mat][0];
      const float hs = 0.5f * scl[t * 2 + mat][1];
      const float hi = is_q ? -hs : hs;          // conj(h) multiplies Q
      const float di0 = mat ? -acc[b][tm][1] : acc[b][tm][1];   // W multiplies conj(x)
      const float di1 = mat ? -acc[b][tm][3] : acc[b][tm][3];
      yr0 = fmaf(hr, acc[b][tm][0], fmaf(-hi, di0, yr0));
      yi0 = fmaf(hr, di0, fmaf(hi, acc[b][tm][0], yi0));
      yr1 = fmaf(hr, acc[b][tm][2], fmaf(-hi, di1, yr1));
      yi1 = fmaf(hr, di1, fmaf(hi, acc[b][tm][2], yi1));
    }
    const float us = t4 < 2 ? -invS[b] : -invS[b] * 0.015625f;  // minus: P = C - P_D
    yr0 *= us; yi0 *= us; yr1 *= us; yi1 *= us;
#pragma unroll
    for (int h = 2; h >= 1; h >>= 1) {
      yr0 += __shfl_xor_sync(0xffffffffu, yr0, h);
      yi0 += __shfl_xor_sync(0xffffffffu, yi0, h);
      yr1 += __shfl_xor_sync(0xffffffffu, yr1, h);
      yi1 += __shfl_xor_sync(0xffffffffu, yi1, h);
    }
    if (t4 == 0) {
      const float ycr = sre_u * cre + sre_w * cre, yci = sre_u * cim - sre_w * cim;
      float* r = red + ((warp * NB + b) * kRows) * 2;
      r[g * 2 + 0] = yr0 + ycr; r[g * 2 + 1] = yi0 + yci;
      r[(g + 8) * 2 + 0] = yr1 + ycr; r[(g + 8) * 2 + 1] = yi1 + yci;
    }
  }
  __syncthreads();
  if (tid < kRows * NB * 2) {
    const int comp = tid & 1, r = (tid >> 1) & 15, b = tid >> 5;
    float sum = 0.f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) sum += red[((w * NB + b) * kRows + r) * 2 + comp];
    const int64_t j = j0 + r;
    if (ok && j < a.n && b < a.B) {
      float* yb = a.y[lin] + (int64_t)b * a.ldy;
      if (comp == 0) yb[j] = sum;
      else if (a.n + j < a.out_features) yb[a.n + j] = sum;
    }
  }
  if (!ok && lane == 0) {
    // Let any copy still in flight land before the CTA's shared memory is released.
    mbar_wait_bounded(bar, 0, kWaitLimit);
  }
}

struct Layout {
  int x_off, raw_off, red_off, bar_off, total;
};

inline Layout layout(int nchunks, int T, int NB) {
  Layout L;
  const int cpw = (nchunks + kWarps - 1) / kWarps;
  L.x_off = nchunks * 2 * T * kTileBytes;
  L.raw_off = L.x_off + kWarps * cpw * NB * kXBytes;
  L.red_off = L.raw_off + kWarps * cpw * NB * 512;
  L.bar_off = L.red_off + kWarps * NB * kRows * 2 * 4;
  L.total = L.bar_off + kWarps * 8;
  return L;
}

template <int NB, int T>
fairy2i_status launch(Args a, int count, const Layout& L, cudaStream_t stream) {
  auto kern = wl_decode_fp8_kernel<NB, T>;
  static std::atomic<uint64_t> smem_set{0};
  if (!smem_attr_once(kern, kMaxSmem, smem_set)) return FAIRY2I_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(a.tiles * count));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = L.total;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, kern, a) != cudaSuccess) return FAIRY2I_ERR_CUDA;
  return FAIRY2I_OK;
}

}  // namespace dec

// `count` linears of the same shape sharing x (codes[g], scales[g] -> y[g]) in one launch.
fairy2i_status launch_wl_decode_group(const void* x, fairy2i_dtype xdt, int64_t B,
                                      int64_t in_features, int64_t ldx, int count,
                                      const uint32_t* const* codes, const float* const* scales,
                                      int64_t n, int64_t m, int64_t out_features, int64_t wpr,
                                      int T, float* const* y, int64_t ldy, cudaStream_t stream,
                                      bool* handled) {
  using namespace dec;
  *handled = false;
  if (xdt != FAIRY2I_BF16 || B > 2 || T > 4 || count < 1 || count > kMaxGroup) return FAIRY2I_OK;
  const int nchunks = (int)(wpr / kChunkWords);
  const int NB = B > 1 ? 2 : 1;
  const Layout L = layout(nchunks, T, NB);
  if (L.total > kMaxSmem || m > (1 << 24) || (nchunks + kWarps - 1) / kWarps > kMaxChunksPerWarp)
    return FAIRY2I_OK;
  Args a;
  for (int g = 0; g < kMaxGroup; ++g) {
    a.codes[g] = codes[g < count ? g : 0];
    a.scales[g] = scales[g < count ? g : 0];
    a.y[g] = y[g < count ? g : 0];
  }
  a.x = reinterpret_cast<const __nv_bfloat16*>(x);
  a.B = B; a.in_features = in_features; a.ldx = ldx;
  a.n = n; a.m = m; a.out_features = out_features; a.ldy = ldy;
  a.wpr = (int)wpr; a.nchunks = nchunks; a.status = device_status_word();
  a.tiles = (int)((n + kRows - 1) / kRows);
  a.x_off = L.x_off; a.raw_off = L.raw_off; a.red_off = L.red_off; a.bar_off = L.bar_off;
  a.cpw = (nchunks + kWarps - 1) / kWarps;
  a.x_vec = (reinterpret_cast<uintptr_t>(x) % 16 == 0) && (ldx % 8 == 0) && (m % 8 == 0);
  *handled = true;
  switch (T * 4 + NB) {
    case 1 * 4 + 1: return launch<1, 1>(a, count, L, stream);
    case 1 * 4 + 2: return launch<2, 1>(a, count, L, stream);
    case 2 * 4 + 1: return launch<1, 2>(a, count, L, stream);
    case 2 * 4 + 2: return launch<2, 2>(a, count, L, stream);
    case 3 * 4 + 1: return launch<1, 3>(a, count, L, stream);
    case 3 * 4 + 2: return launch<2, 3>(a, count, L, stream);
    case 4 * 4 + 1: return launch<1, 4>(a, count, L, stream);
    case 4 * 4 + 2: return launch<2, 4>(a, count, L, stream);
  }
  *handled = false;
  return FAIRY2I_OK;
}

fairy2i_status launch_wl_decode(const void* x, fairy2i_dtype xdt, int64_t B, int64_t in_features,
                                int64_t ldx, const uint32_t* codes, const float* scales,
                                int64_t n, int64_t m, int64_t out_features, int64_t wpr, int T,
                                float* y, int64_t ldy, cudaStream_t stream, bool* handled) {
  return launch_wl_decode_group(x, xdt, B, in_features, ldx, 1, &codes, &scales, n, m,
                                out_features, wpr, T, &y, ldy, stream, handled);
}

}  // namespace fairy2i
