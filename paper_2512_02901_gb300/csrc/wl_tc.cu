// Decode (B <= 2 tokens) kernel of the quantized widely-linear matmul on the 5th-generation
// tensor cores (tcgen05.mma with the code matrix in tensor memory).
//
// Arithmetic (Eq. ifairy-dequant, Algorithm 1 with the W conj(x) term): every code carries the
// signs sigma = sign(Re b + Im b), tau = sign(Re b - Im b) of its codeword b, and with
// h = (s_re + i s_im)/2 the dequantized weight is h sigma + conj(h) tau. Per (stage t, matrix)
// the layer needs P = sum_k sigma_k x_k and Q = sum_k tau_k x_k for every output row; then
// y += h P + conj(h) Q for U and h conj(P) + conj(h) conj(Q) for W.
//
// Tensor-core form. One tcgen05.mma (M = 128, N = 16, K = 32, e4m3 x e4m3 -> f32) covers one
// code word (16 codes) of 128 (stage-matrix, row) pairs: TMEM lane tm*R + r holds row r of
// stage-matrix tm (tm = 2 t + matrix, R = 64, 32, 16, 16 rows for T = 1..4). The word is
// decoded into the 32 A bytes (sigma and tau planes of its 16 codes) by one LOP3 per 4 bytes,
// each byte an e4m3 value affine in its bit (a = alpha + 2 bit, sigma = (1 + alpha) - a), so
// P = C - D with D the MMA result and C = sum_k (1 + alpha_k) x_k shared by all rows. B holds
// x split exactly into two e4m3 limbs (hi = e4m3(x S), lo = e4m3(64 (x S - hi)), S a power of
// two per CTA and token) in the 16 columns (token, limb, sigma/tau slot, re/im).
//
// Work split. A row block (R rows of every stage-matrix) is cut along K into ks contiguous
// ranges of 128-code chunks, one per CTA of a thread-block cluster of ks CTAs (ks = 1: no
// cluster); the cluster sums its partial rows through distributed shared memory in rank order
// (deterministic) and rank 0 writes y. A unit is one chunk of the row block: 8 words, 8 MMAs,
// 4 KB of codes, consecutive in memory for every 16-row tile, so a group of kGU units arrives as
// one bulk copy per tile. One CTA per SM (it holds all 512 TMEM columns), so no CTA ever waits for
// tensor memory held by another.
//
// Roles (21 warps). Warps 0-11 form three sets of four (warp w reaches TMEM lanes 32 (w % 4) ..);
// set d owns units d, d + 3, d + 6, ... and two one-unit A slots in TMEM: its four warps decode a
// unit into a slot, meet at the set's named barrier, and warps 4d, 4d + 1 then issue the MMAs of
// words 0-3 and 4-7 into the set's two accumulators; the slot is written again once those MMAs
// have completed. The sets read only the codes, so they start before the previous kernel in the
// stream has finished. Warp 13 copies the first code group; warp 12 copies (after the
// programmatic-launch wait) this CTA's slice of x, then the other code groups. Warps 13-20 turn x into the B tiles
// of every unit at once, then compute the C term while the MMAs run.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_fp8.h>

#include <mutex>

#include "common.cuh"
#include "ptx.cuh"
#include "tc.cuh"

namespace fairy2i {

namespace tcd {

constexpr int kSets = 3;                           // decode + issue sets of 4 warps
constexpr int kSetWarps = 4 * kSets;               // 12
constexpr int kCopyWarp = kSetWarps;               // 12
constexpr int kXWarp0 = kCopyWarp + 1;             // 13
constexpr int kXWarps = 8;
constexpr int kWarps = kXWarp0 + kXWarps;          // 21
constexpr int kThreads = kWarps * 32;              // 672
constexpr int kXThreads = kXWarps * 32;            // 256
constexpr int kGU = 6;                             // units per code group (one copy per tile)
constexpr int kSG = 3;                             // code group stages
constexpr int kUnitBytes = 4096;                   // 128 lanes x 8 words
constexpr int kSlots = 2;                          // TMEM A slots per set, one unit each
constexpr int kWordB = 512;                        // B tile of one word: 16 rows x 32 bytes
constexpr int kUnitB = 8 * kWordB;                 // B tiles of one unit, 4 KB
constexpr int kMaxUnits = 22;                      // 128-code chunks per CTA
constexpr int kTmemCols = 512;
constexpr int kColA = kSets * 2 * 16;              // D: two 16-column accumulators per set
constexpr int kXsBytes = 2 * 2 * kMaxUnits * 256;  // bf16 x: [token][part][unit][128]
constexpr int kMaxCluster = 8;
constexpr int kPartFloats = 256;                   // one partial: 64 rows x 2 tokens x (re, im)
constexpr uint64_t kWaitNs = 1000000000ull;        // 1 s: a pipeline wait is microseconds
constexpr uint32_t kIdesc = idesc_e4m3_f32(128, 16);
static_assert(kColA + kSets * kSlots * 64 <= kTmemCols, "TMEM columns");

// Shared memory layout (bytes from the 1024-aligned base).
constexpr int kOffCodes = 0;
constexpr int kOffB = kOffCodes + kSG * kGU * kUnitBytes;        // 72 KB
constexpr int kOffXs = kOffB + kMaxUnits * kUnitB;               // + 88 KB
constexpr int kOffC = kOffXs + kXsBytes;                         // + 22 KB
constexpr int kOffDx = kOffC + kMaxUnits * 16;                   // float [22][4]
constexpr int kOffRed = kOffDx + (kSets - 1) * 128 * 16 * 4;     // float [2][16][128]
constexpr int kOffGather = kOffRed + 128 * 2 * 2 * 4;            // float [128][2][2]
constexpr int kOffBar = kOffGather + kMaxCluster * kPartFloats * 4;
constexpr int kNumBars = 2 * kSG + 2 * kSets * kSlots + kSets + 4 + 2 * kSets;
constexpr int kOffMisc = kOffBar + kNumBars * 8;
constexpr int kSmemBytes = kOffMisc + 512 + 1024;                // + alignment slack
static_assert(kSmemBytes > 116 * 1024, "one CTA per SM: it owns all TMEM columns");
static_assert(kSmemBytes <= 227 * 1024, "shared memory per CTA");

struct Args {
  const uint32_t* codes;
  const __nv_bfloat16* x;
  const float* scales;
  float* y;
  unsigned int* status;
  int64_t B, in_features, ldx, n, m, out_features, ldy;
  int nch;        // 128-code chunks per row
  int row_tiles;  // ceil(n / 16)
  int ks;         // CTAs per row block (cluster size)
  int x_vec;      // x rows 16-byte aligned with m % 8 == 0: vector loads allowed
  int x_bulk;     // and in_features even: x slices arrive by bulk copy
};

struct Misc {
  uint32_t tmem;
  int abort;
  float S[2], invS[2];
  float cseg[4];
  unsigned int xmax[2];           // max |x| per token, as float bits
  float scales[4 * 4];            // (s_re, s_im) per stage and matrix
};

// Bounded wait that gives up at once when another role has already given up.
__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, volatile int* abort,
                                              unsigned int* status) {
  if (*abort) return false;
  if (mbar_wait_timed(bar, parity, kWaitNs)) return true;
  *abort = 1;
  latch_status(status, kStatusTimeout);
  return false;
}

// A register j (0..7) of a word: e4m3 bytes (sigma_2j, sigma_2j+1, tau_2j, tau_2j+1), each
// alpha_q + 2 bit with q the bit position used (2, 3, 2, 3, 6, 7, 6, 7 for j = 0..7; words
// shifted left by 2 for j in {0, 1, 4, 5}); 1 + alpha = 5, 3, 5, 3, 1, 0, 1, 0.
__device__ __forceinline__ void decode_word(uint32_t w0, uint32_t* r) {
  const uint32_t w2 = w0 << 2;
  r[0] = lop3_and_or(w2, 0x04040404u, 0x48484848u);   // q = 2: 4 + 2 bit
  r[1] = lop3_and_or(w2, 0x08080808u, 0x40404040u);   // q = 3: 2 + 2 bit
  r[2] = lop3_and_or(w0, 0x04040404u, 0x48484848u);
  r[3] = lop3_and_or(w0, 0x08080808u, 0x40404040u);
  r[4] = w2 & 0x40404040u;                            // q = 6: 0 + 2 bit
  r[5] = lop3_and_xor(w2, 0x80808080u, 0xB8B8B8B8u);  // q = 7: -1 + 2 bit
  r[6] = w0 & 0x40404040u;
  r[7] = lop3_and_xor(w0, 0x80808080u, 0xB8B8B8B8u);
}

__device__ __forceinline__ float bf_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

__device__ __forceinline__ uint32_t e4m3x2(float a, float b) {
  return (uint32_t)__nv_cvt_float2_to_fp8x2(make_float2(a, b), __NV_SATFINITE, __NV_E4M3);
}
__device__ __forceinline__ float2 e4m3x2_to_float2(uint32_t v) {
  return __half22float2(
      __half2(__nv_cvt_fp8x2_to_halfraw2((__nv_fp8x2_storage_t)v, __NV_E4M3)));
}

// Power-of-two S with max|x| S < 128, and 1/S, from the exponent bits of max|x|.
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

// Row n of a word's B tile, K bytes 16 hh .. 16 hh + 15 (core matrices of 8 rows x 16 bytes,
// K-adjacent at +128, 8-row groups at +256).
__device__ __forceinline__ void store_brow(unsigned char* tile, int n, int hh, uint4 v) {
  *reinterpret_cast<uint4*>(tile + (n >> 3) * 256 + hh * 128 + (n & 7) * 16) = v;
}

// Eight bf16 values of part `part` (0 = re, 1 = im) of token b at complex index k (k % 8 == 0),
// zero outside the valid range of that part.
__device__ __forceinline__ uint4 load_x8(const Args& a, int b, int part, int64_t k) {
  const __nv_bfloat16* row = a.x + (int64_t)b * a.ldx + (int64_t)part * a.m;
  const int64_t lim = part ? a.in_features - a.m : a.m;
  if (a.x_vec && k + 8 <= lim) return __ldg(reinterpret_cast<const uint4*>(row + k));
  uint32_t w[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t k0 = k + 2 * i, k1 = k0 + 1;
    const uint32_t lo = k0 < lim ? (uint32_t)__bfloat16_as_ushort(row[k0]) : 0u;
    const uint32_t hi = k1 < lim ? (uint32_t)__bfloat16_as_ushort(row[k1]) : 0u;
    w[i] = lo | (hi << 16);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

template <int NB, int T>
__global__ void __launch_bounds__(kThreads, 1) wl_tc_decode_kernel(const Args a) {
  constexpr int TM = 2 * T;
  constexpr int R = (T == 1) ? 64 : (T == 2 ? 32 : 16);  // rows per row block
  constexpr int RT = R / 16;                              // 16-row code tiles per row block
  constexpr int NV = R * NB * 2;                          // outputs of a row block
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kOffBar);
  uint64_t* cfull = bars;                       // code group landed         (tx count)
  uint64_t* cempty = cfull + kSG;               // code group read            (4 warps x kGU units)
  uint64_t* sfull = cempty + kSG;               // [set][slot] A slot written  (4 warps)
  uint64_t* sfree = sfull + kSets * kSlots;     // [set][slot] its MMAs done   (2 issuer commits)
  uint64_t* sdone = sfree + kSets * kSlots;     // [set] every MMA of the set  (2 issuer commits)
  uint64_t* xfull = sdone + kSets;              // x slice landed             (tx count)
  uint64_t* bready = xfull + 1;                 // every B tile written       (1 arrival)
  uint64_t* cready = bready + 1;                // C term written             (1 arrival)
  uint64_t* gbar = cready + 1;                  // rank 0: partials of the other ranks arrived
  uint64_t* fin = gbar + 1;                     // [set][issuer]: abort path
  Misc* misc = reinterpret_cast<Misc*>(smem + kOffMisc);
  volatile int* abort_flag = &misc->abort;
  __nv_bfloat16* xs = reinterpret_cast<__nv_bfloat16*>(smem + kOffXs);  // [b][p][unit*128]
  float* Cch = reinterpret_cast<float*>(smem + kOffC);
  float* dx = reinterpret_cast<float*>(smem + kOffDx);
  float* red = reinterpret_cast<float*>(smem + kOffRed);
  float* gather = reinterpret_cast<float*>(smem + kOffGather);

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int ks = a.ks;
  const int rank = ks > 1 ? (int)cluster_ctarank() : 0;
  const int rb = (int)(blockIdx.x / (unsigned)ks);
  const int c0 = (rank * a.nch) / ks;
  const int units = ((rank + 1) * a.nch) / ks - c0;
  const int ngroups = (units + kGU - 1) / kGU;
  int ntiles = 0;   // existing 16-row tiles of this row block
#pragma unroll
  for (int rt = 0; rt < RT; ++rt) ntiles += (rb * RT + rt < a.row_tiles) ? 1 : 0;

  // ---- prologue: barriers, TMEM ----
  if (tid == 0) {
    for (int i = 0; i < kSG; ++i) {
      mbar_init(&cfull[i], 1);
      mbar_init(&cempty[i], 4 * kGU);
    }
    for (int i = 0; i < kSets * kSlots; ++i) {
      mbar_init(&sfull[i], 4);
      mbar_init(&sfree[i], 2);
    }
    for (int i = 0; i < kSets; ++i) mbar_init(&sdone[i], 2);
    mbar_init(xfull, 1);
    mbar_init(bready, 1);
    mbar_init(cready, 1);
    mbar_init(gbar, ks > 1 ? (ks - 1) * 4 * 32 : 1);
    for (int i = 0; i < 2 * kSets; ++i) mbar_init(&fin[i], 1);
    misc->abort = 0;
    misc->xmax[0] = misc->xmax[1] = 0u;
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&misc->tmem, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (ks > 1) cluster_arrive();   // barriers of every rank initialised (waited before DSMEM use)
  const uint32_t tmem = misc->tmem;

  // Code group g (units kGU g ..) into stage g % kSG, laid out [tile tm*RT + rt][unit][512 B]:
  // one bulk copy per existing tile, issued by lanes 0 .. TM*RT-1 of the calling warp.
  auto issue_group = [&](int g) {
    const int nu = min(kGU, units - g * kGU);
    uint64_t* bar = &cfull[g % kSG];
    if (lane == 0) mbar_arrive_expect_tx(bar, (uint32_t)(TM * ntiles * nu * 512));
    __syncwarp();
    const int tm = lane / RT, rt = lane % RT;
    if (lane < TM * RT && rt < ntiles) {
      const int64_t tile = (int64_t)tm * a.row_tiles + rb * RT + rt;
      bulk_load(smem + kOffCodes + (g % kSG) * kGU * kUnitBytes + (lane * kGU) * 512,
                a.codes + (tile * a.nch + c0 + g * kGU) * 128, (uint32_t)(nu * 512), bar);
    }
  };
  if (warp == kXWarp0 && ngroups > 0) issue_group(0);   // the copy warp takes x first
  pdl_launch_dependents();

  if (warp < kSetWarps) {
    // ------------- sets: decode a unit into a slot, then two warps issue its MMAs -------------
    const int set = warp >> 2, quarter = warp & 3;
    const int L = quarter * 32 + lane;
    const uint32_t codes_addr =
        smem_u32(smem + kOffCodes) + (uint32_t)((L >> 4) * kGU * 512 + (L & 15) * 32);
    const uint32_t t_lane = tmem + ((uint32_t)(quarter * 32) << 16) + kColA;
    int j = 0;
    // Software pipeline: the A stores of unit j are announced once the first half of unit j + 1
    // is decoded (the store wait then finds them done).
    int pend = -1;          // slot written but not yet announced
    bool ok = true;
    for (int u = set; u < units; u += kSets, ++j) {
      const int sl = j % kSlots, g = u / kGU, ui = u - g * kGU, st = g % kSG;
      const int si = set * kSlots + sl;
      ok = __all_sync(0xffffffffu, wait_or_abort(&cfull[st], (g / kSG) & 1, abort_flag, a.status));
      if (!ok) break;
      const uint32_t src = codes_addr + st * kGU * kUnitBytes + ui * 512;
      const uint4 q0 = lds128(src), q1 = lds128(src + 16);
      const uint32_t a_col = t_lane + si * 64;
      uint32_t r[32];
      decode_word(q0.x, r);
      decode_word(q0.y, r + 8);
      decode_word(q0.z, r + 16);
      decode_word(q0.w, r + 24);
      __syncwarp();
      if (lane == 0) mbar_arrive(&cempty[st]);
      if (pend >= 0) {
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sfull[pend]);
        pend = -1;
      }
      if (j >= kSlots)   // the slot's previous unit has been consumed
        ok = __all_sync(0xffffffffu, wait_or_abort(&sfree[si], ((j / kSlots) - 1) & 1, abort_flag,
                                                   a.status));
      if (!ok) break;
      tmem_st32(a_col, r);
      decode_word(q1.x, r);
      decode_word(q1.y, r + 8);
      decode_word(q1.z, r + 16);
      decode_word(q1.w, r + 24);
      tmem_st32(a_col + 32, r);
      pend = si;
    }
    if (ok && pend >= 0) {
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sfull[pend]);
    }

    // ---- epilogue: each warp sums its set's two accumulators for its 32 lanes ----
    float d[16];
#pragma unroll
    for (int k = 0; k < 16; ++k) d[k] = 0.f;
    const bool done = set * 1 < units &&
                      __all_sync(0xffffffffu, wait_or_abort(&sdone[set], 0, abort_flag, a.status));
    if (done) {
      tc_fence_after();
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        float v[16];
        tmem_ld16(tmem + ((uint32_t)(quarter * 32) << 16) + (set * 2 + e) * 16, v);
        tmem_wait_ld();
#pragma unroll
        for (int k = 0; k < 16; ++k) d[k] += v[k];
      }
    }
    tc_fence_before();
    if (set > 0) {
#pragma unroll
      for (int k = 0; k < 16; ++k) dx[((set - 1) * 16 + k) * 128 + L] = d[k];
    }
    named_bar_sync(1, kSetWarps * 32);
    if (set == 0) {
#pragma unroll
      for (int k = 0; k < 16; ++k) d[k] += dx[k * 128 + L] + dx[(16 + k) * 128 + L];
      (void)__all_sync(0xffffffffu, wait_or_abort(cready, 0, abort_flag, a.status));
      if (L < TM * R) {
        const int tm = L / R;
        const float hr = 0.5f * misc->scales[tm * 2 + 0];
        const float hi = 0.5f * misc->scales[tm * 2 + 1];
        const bool mat = tm & 1;
#pragma unroll
        for (int b = 0; b < NB; ++b) {
          const float cre = misc->cseg[b * 2 + 0], cim = misc->cseg[b * 2 + 1];
          const float is = misc->invS[b];
          // column (token, limb, slot, part) = ((b 2 + limb) 2 + slot) 2 + part
          const int c = b * 8;
          const float pre = cre - (d[c + 0] + 0.015625f * d[c + 4]) * is;
          float pim = cim - (d[c + 1] + 0.015625f * d[c + 5]) * is;
          const float qre = cre - (d[c + 2] + 0.015625f * d[c + 6]) * is;
          float qim = cim - (d[c + 3] + 0.015625f * d[c + 7]) * is;
          if (mat) {                 // W multiplies conj(x): conjugate P and Q
            pim = -pim;
            qim = -qim;
          }
          red[(L * NB + b) * 2 + 0] = hr * pre - hi * pim + hr * qre + hi * qim;
          red[(L * NB + b) * 2 + 1] = hr * pim + hi * pre + hr * qim - hi * qre;
        }
      }
      named_bar_sync(2, 4 * 32);
      // Sum over the stage-matrices: value idx = (row rr, token b, re/im).
      float vals[(NV + 127) / 128];
#pragma unroll
      for (int it = 0; it < (NV + 127) / 128; ++it) {
        const int idx = L + it * 128;
        float sum = 0.f;
        if (idx < NV) {
          const int rr = idx / (NB * 2), rest = idx % (NB * 2);
#pragma unroll
          for (int m2 = 0; m2 < TM; ++m2) sum += red[(m2 * R + rr) * NB * 2 + rest];
        }
        vals[it] = sum;
      }
      if (ks > 1) {
        cluster_wait();                // every rank's barriers are initialised
        if (rank != 0) {
          const uint32_t g0 = smem_u32(gather);
#pragma unroll
          for (int it = 0; it < (NV + 127) / 128; ++it) {
            const int idx = L + it * 128;
            if (idx < NV)
              st_cluster_f32(mapa_shared(g0 + (rank * kPartFloats + idx) * 4, 0), vals[it]);
          }
          mbar_arrive_remote(mapa_shared(smem_u32(gbar), 0));
        } else {
          const bool got = __all_sync(0xffffffffu, !*abort_flag &&
                                                       mbar_wait_cluster_timed(gbar, 0, kWaitNs));
          if (!got) {
            *abort_flag = 1;
            latch_status(a.status, kStatusTimeout);
          } else {
#pragma unroll
            for (int it = 0; it < (NV + 127) / 128; ++it) {
              const int idx = L + it * 128;
              if (idx < NV)
                for (int r2 = 1; r2 < ks; ++r2) vals[it] += gather[r2 * kPartFloats + idx];
            }
          }
        }
      }
      if (rank == 0 && !*abort_flag) {
#pragma unroll
        for (int it = 0; it < (NV + 127) / 128; ++it) {
          const int idx = L + it * 128;
          if (idx < NV) {
            const int rr = idx / (NB * 2), b = (idx >> 1) % NB, comp = idx & 1;
            const int64_t jr = (int64_t)rb * R + rr;
            if (b < a.B && jr < a.n) {
              float* yb = a.y + (int64_t)b * a.ldy;
              if (comp == 0) yb[jr] = vals[it];
              else if (a.n + jr < a.out_features) yb[a.n + jr] = vals[it];
            }
          }
        }
      }
    }
  } else if (warp == kCopyWarp) {
    // ---------------- copies: x slice (after the programmatic wait), then the codes ----------
    if (a.x_bulk && lane < 2 * NB && lane / 2 < a.B) {
      // Warm L2 with this CTA's x slice; the copy below (after the wait) reads the final values.
      const int b = lane >> 1, p = lane & 1;
      const int64_t lim = p ? a.in_features - a.m : a.m;
      const int64_t k0 = (int64_t)c0 * 128, k1 = min((int64_t)(c0 + units) * 128, lim);
      if (k1 > k0)
        prefetch_l2_bulk(a.x + (int64_t)b * a.ldx + (int64_t)p * a.m + k0, (uint32_t)((k1 - k0) * 2));
    }
    pdl_wait_primary();   // x may be written by the previous kernel
    if (a.x_bulk) {
      // per (token, part): complex indices [c0 128, min((c0 + units) 128, lim)) of the row
      uint32_t total = 0, mine = 0;
#pragma unroll
      for (int jx = 0; jx < 2 * NB; ++jx) {
        const int b = jx >> 1, p = jx & 1;
        const int64_t lim = p ? a.in_features - a.m : a.m;
        const int64_t k0 = (int64_t)c0 * 128, k1 = min((int64_t)(c0 + units) * 128, lim);
        const uint32_t by = (b < a.B && k1 > k0) ? (uint32_t)((k1 - k0) * 2) : 0u;
        total += by;
        if (lane == jx) mine = by;
      }
      if (lane == 0) mbar_arrive_expect_tx(xfull, total);
      __syncwarp();
      if (lane < 2 * NB && mine > 0) {
        const int b = lane >> 1, p = lane & 1;
        bulk_load(xs + (b * 2 + p) * kMaxUnits * 128,
                  a.x + (int64_t)b * a.ldx + (int64_t)p * a.m + (int64_t)c0 * 128, mine, xfull);
      }
    }
    for (int g = 1; g < ngroups && g < kSG; ++g) issue_group(g);
    // Refill a group stage once it has been decoded.
    for (int g = kSG; g < ngroups; ++g) {
      const int gp = g - kSG;
      const bool free = lane != 0 ||
                        wait_or_abort(&cempty[gp % kSG], (gp / kSG) & 1, abort_flag, a.status);
      if (!__all_sync(0xffffffffu, free)) break;
      issue_group(g);
    }
    // Abort path: let every issued copy land before shared memory is released.
    if (lane == 0 && *abort_flag) {
      for (int g = 0; g < ngroups; ++g)
        (void)mbar_wait_timed(&cfull[g % kSG], (g / kSG) & 1, 1000000ull);
      if (a.x_bulk) (void)mbar_wait_timed(xfull, 0, 1000000ull);
    }
  } else {
    // ---------------- warps 13-20: x -> B tiles of every unit, then the C term ----------------
    pdl_wait_primary();   // x may be written by the previous kernel
    const int xt = tid - kXWarp0 * 32;   // 0 .. kXThreads-1
    if (xt < TM * 2) misc->scales[xt] = __ldg(a.scales + xt);
    if (a.x_bulk) {
      // zero what the copy does not cover: values past the end of the row
      for (int q = xt; q < 2 * NB * units * 16; q += kXThreads) {
        const int v = q % (units * 16), p = (q / (units * 16)) & 1, b = q / (units * 32);
        const int64_t lim = p ? a.in_features - a.m : a.m;
        if (b >= a.B || (int64_t)c0 * 128 + v * 8 >= lim)
          *reinterpret_cast<uint4*>(xs + (b * 2 + p) * kMaxUnits * 128 + v * 8) =
              make_uint4(0, 0, 0, 0);
      }
      (void)__all_sync(0xffffffffu, wait_or_abort(xfull, 0, abort_flag, a.status));
    } else {
      for (int q = xt; q < 2 * NB * units * 16; q += kXThreads) {
        const int v = q % (units * 16), p = (q / (units * 16)) & 1, b = q / (units * 32);
        const uint4 u4 = b < a.B ? load_x8(a, b, p, (int64_t)c0 * 128 + v * 8)
                                 : make_uint4(0, 0, 0, 0);
        *reinterpret_cast<uint4*>(xs + (b * 2 + p) * kMaxUnits * 128 + v * 8) = u4;
      }
    }
    named_bar_sync(3, kXThreads);
    // max |x| per token (float bits of non-negative values order like unsigned integers)
    {
      unsigned int mx0 = 0u, mx1 = 0u;
      for (int q = xt; q < 2 * NB * units * 16; q += kXThreads) {
        const int v = q % (units * 16), p = (q / (units * 16)) & 1, b = q / (units * 32);
        const uint4 u4 = *reinterpret_cast<const uint4*>(xs + (b * 2 + p) * kMaxUnits * 128 + v * 8);
        const uint32_t e[4] = {u4.x, u4.y, u4.z, u4.w};
        unsigned int m8 = 0u;
#pragma unroll
        for (int i = 0; i < 4; ++i)
          m8 = max(m8, max((e[i] << 17) >> 1, (e[i] & 0x7fff0000u)));   // |bf16| as f32 bits
        if (b == 0) mx0 = max(mx0, m8); else mx1 = max(mx1, m8);
      }
      const unsigned int w0 = __reduce_max_sync(0xffffffffu, mx0);
      const unsigned int w1 = __reduce_max_sync(0xffffffffu, mx1);
      if (lane == 0) {
        atomicMax(&misc->xmax[0], w0);
        if (NB > 1) atomicMax(&misc->xmax[1], w1);
      }
    }
    named_bar_sync(3, kXThreads);
    float S[2], invS[2];
#pragma unroll
    for (int b = 0; b < NB; ++b) pow2_scale(__uint_as_float(misc->xmax[b]), S[b], invS[b]);
    if (xt < NB) misc->invS[xt] = invS[xt];
    // B tiles: task (unit, token, word, half, row): one 16-byte row half per lane, the eight lanes
    // of a shared-memory phase writing the eight rows of one core matrix (no bank conflicts).
    // Row n = ((b 2 + limb) 2 + slot) 2 + p holds the limb bytes of codes 2j', 2j'+1 in the sigma
    // half (bytes 0-1) or the tau half (bytes 2-3) of register j'. The eight lanes of a row group
    // convert the 16 values of the group once (lane nl: values 2 (nl & 3), + 1 of part nl >> 2)
    // and exchange the limb pairs by shuffles.
    for (int q = xt; q < NB * units * 128; q += kXThreads) {   // warp-uniform: multiples of 32
      const int nl = q & 7, hh = (q >> 3) & 1, wd = (q >> 4) & 7, rest = q >> 7;
      const int b = rest % NB, u = rest / NB;
      const int limb = nl >> 2, slot = (nl >> 1) & 1, p = nl & 1;
      const uint32_t e2 = *reinterpret_cast<const uint32_t*>(
          xs + (b * 2 + (nl >> 2)) * kMaxUnits * 128 + u * 128 + wd * 16 + hh * 8 + 2 * (nl & 3));
      const float v0 = bf_lo(e2) * S[b], v1 = bf_hi(e2) * S[b];
      const uint32_t hp = e4m3x2(v0, v1) & 0xffffu;
      const float2 hf = e4m3x2_to_float2(hp);
      const uint32_t lp = e4m3x2(64.f * (v0 - hf.x), 64.f * (v1 - hf.y)) & 0xffffu;
      const uint32_t both = hp | (lp << 16);
      uint32_t w[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const uint32_t v = __shfl_sync(0xffffffffu, both, (lane & ~7) | (p * 4 + i));
        w[i] = (limb ? (v >> 16) : (v & 0xffffu)) << (slot ? 16 : 0);
      }
      store_brow(smem + kOffB + u * kUnitB + wd * kWordB, b * 8 + nl, hh,
                 make_uint4(w[0], w[1], w[2], w[3]));
    }
    fence_proxy_async_smem();
    named_bar_sync(3, kXThreads);
    if (xt == 0) mbar_arrive(bready);
    const int xw = warp - kXWarp0;
    if (xw < 2 * kSets) {
      // ------ MMA issuers: lane 0 of x-warp 2 d + e issues words 4 e .. 4 e + 3 of every unit of
      // set d (its own accumulator), once the set's four warps have written the unit ------
      const int set = xw >> 1, e = xw & 1;
      if (lane == 0) {
        const uint32_t d_tmem = tmem + (set * 2 + e) * 16;
        const uint32_t b_base = smem_u32(smem + kOffB);
        bool issued = false;
        int j = 0;
        for (int u = set; u < units; u += kSets, ++j) {
          const int si = set * kSlots + j % kSlots;
          if (!wait_or_abort(&sfull[si], (j / kSlots) & 1, abort_flag, a.status)) break;
          tc_fence_after();
          const uint32_t a_slot = tmem + kColA + si * 64;
#pragma unroll
          for (int w4 = 0; w4 < 4; ++w4) {
            const int wd = e * 4 + w4;
            mma_e4m3_ts(d_tmem, a_slot + wd * 8,
                        smem_desc(b_base + u * kUnitB + wd * kWordB, 128, 256), kIdesc,
                        (j > 0 || w4 > 0) ? 1u : 0u);
          }
          issued = true;
          mma_commit(&sfree[si]);
          if (u + kSets >= units) mma_commit(&sdone[set]);
        }
        // Abort path: MMAs this thread issued must finish before TMEM is released.
        if (issued && *abort_flag) {
          mma_commit(&fin[set * 2 + e]);
          (void)mbar_wait_timed(&fin[set * 2 + e], 0, kWaitNs);
        }
      }
      __syncwarp();
    } else {
      // ------ the other x-warps: C term (needed by the epilogue only) ------
      constexpr int kCThreads = kXThreads - 2 * kSets * 32;
      const int ct = xt - 2 * kSets * 32;   // 0 .. kCThreads-1
      // task (token, chunk, part, 8 values)
      for (int q = ct; q < NB * units * 32; q += kCThreads) {   // warp-uniform: multiples of 32
        const int v = q & 15, p = (q >> 4) & 1, lc = (q >> 5) % units, b = (q >> 5) / units;
        const uint4 u4 =
            *reinterpret_cast<const uint4*>(xs + (b * 2 + p) * kMaxUnits * 128 + lc * 128 + v * 8);
        const uint32_t e[4] = {u4.x, u4.y, u4.z, u4.w};
        // 1 + alpha of codes 8h .. 8h + 7 of a word (h = v & 1): 5,5,3,3,5,5,3,3 or 1,1,0,0,..
        const float p0 = bf_lo(e[0]) + bf_hi(e[0]), p1 = bf_lo(e[1]) + bf_hi(e[1]);
        const float p2 = bf_lo(e[2]) + bf_hi(e[2]), p3 = bf_lo(e[3]) + bf_hi(e[3]);
        float cs = (v & 1) ? (p0 + p2) : (5.f * (p0 + p2) + 3.f * (p1 + p3));
#pragma unroll
        for (int h = 8; h >= 1; h >>= 1) cs += __shfl_xor_sync(0xffffffffu, cs, h);
        if (v == 0) Cch[lc * 4 + b * 2 + p] = cs;
      }
      named_bar_sync(4, kCThreads);
      if (ct < 2 * NB) {
        float cs = 0.f;
#pragma unroll 1
        for (int lc = 0; lc < units; ++lc) cs += Cch[lc * 4 + ct];
        misc->cseg[ct] = cs;
      }
      named_bar_sync(4, kCThreads);
      if (ct == 0) mbar_arrive(cready);
    }
  }

  // Every thread pairs its cluster arrive (set 0 waited in the epilogue). Rank 0 leaves only after
  // the partials of every other rank have arrived, so no CTA writes into a CTA that left.
  if (ks > 1 && warp >= 4) cluster_wait();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0) tmem_dealloc(tmem, kTmemCols);
}

template <int NB, int T>
fairy2i_status launch(const Args& a, int64_t grid, cudaStream_t stream) {
  auto kern = wl_tc_decode_kernel<NB, T>;
  static std::atomic<uint64_t> smem_set{0};
  if (!smem_attr_once(kern, kSmemBytes, smem_set)) return FAIRY2I_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = (unsigned)a.ks;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  if (cudaLaunchKernelEx(&cfg, kern, a) != cudaSuccess) return FAIRY2I_ERR_CUDA;
  return FAIRY2I_OK;
}

}  // namespace tcd

namespace {
std::mutex g_sm_mu;
int g_sm_count[64];
}  // namespace

static int sm_count(int dev) {
  std::lock_guard<std::mutex> lock(g_sm_mu);
  if (!g_sm_count[dev]) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    g_sm_count[dev] = v;
  }
  return g_sm_count[dev];
}

// CTAs per row block (cluster size, 1..8): the smallest value that keeps a CTA's chunks within
// kMaxUnits, then the one that minimises the estimated time, waves x (fixed cost + units per CTA),
// with the fixed cost of a CTA (prologue, x staging, epilogue) worth about kFixedUnits units.
int wl_tc_cluster_size(int64_t row_blocks, int64_t nch, int sms) {
  const int64_t max_units = tcd::kMaxUnits;
  constexpr int64_t kFixedUnits = 15;
  if (row_blocks < 1 || nch < 1 || sms < 1) return 0;
  const int64_t need = (nch + max_units - 1) / max_units;
  if (need > tcd::kMaxCluster) return 0;
  int best = (int)need;
  int64_t best_cost = -1;
  for (int64_t ks = need; ks <= tcd::kMaxCluster && ks <= nch; ++ks) {
    const int64_t waves = (row_blocks * ks + sms - 1) / sms;
    const int64_t cost = waves * (kFixedUnits + (nch + ks - 1) / ks);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = (int)ks;
    }
  }
  return best;
}

// Handles B <= 2 bf16 tokens, T <= 4 and rows of at most 8 kMaxUnits 128-code chunks; anything
// else is left to the other kernels (*handled = false).
fairy2i_status launch_wl_tc(const void* x, fairy2i_dtype xdt, int64_t B, int64_t in_features,
                            int64_t ldx, const uint32_t* codes, const float* scales, int64_t n,
                            int64_t m, int64_t out_features, int64_t wpr, int T, float* y,
                            int64_t ldy, cudaStream_t stream, bool* handled) {
  using namespace tcd;
  *handled = false;
  if (xdt != FAIRY2I_BF16 || B > 2 || T > 4) return FAIRY2I_OK;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return FAIRY2I_ERR_CUDA;
  const int sms = sm_count(dev);
  if (sms < 1) return FAIRY2I_ERR_CUDA;
  const int NB = B > 1 ? 2 : 1;
  const int R = T == 1 ? 64 : (T == 2 ? 32 : 16);
  const int64_t row_blocks = (n + R - 1) / R;
  const int64_t nch = wpr / 8;
  const int ks = wl_tc_cluster_size(row_blocks, nch, sms);
  if (ks < 1 || row_blocks * ks > (int64_t(1) << 31) - 1 || nch * tcd::kMaxCluster > (1 << 30))
    return FAIRY2I_OK;
  Args a;
  a.codes = codes;
  a.x = reinterpret_cast<const __nv_bfloat16*>(x);
  a.scales = scales;
  a.y = y;
  a.status = device_status_word();
  a.B = B; a.in_features = in_features; a.ldx = ldx; a.n = n; a.m = m;
  a.out_features = out_features; a.ldy = ldy;
  a.nch = (int)nch; a.row_tiles = (int)((n + 15) / 16); a.ks = ks;
  a.x_vec = (reinterpret_cast<uintptr_t>(x) % 16 == 0) && (ldx % 8 == 0) && (m % 8 == 0);
  a.x_bulk = a.x_vec && (in_features % 2 == 0);
  const int64_t grid = row_blocks * ks;
  *handled = true;
  switch (T * 4 + NB) {
    case 1 * 4 + 1: return launch<1, 1>(a, grid, stream);
    case 1 * 4 + 2: return launch<2, 1>(a, grid, stream);
    case 2 * 4 + 1: return launch<1, 2>(a, grid, stream);
    case 2 * 4 + 2: return launch<2, 2>(a, grid, stream);
    case 3 * 4 + 1: return launch<1, 3>(a, grid, stream);
    case 3 * 4 + 2: return launch<2, 3>(a, grid, stream);
    case 4 * 4 + 1: return launch<1, 4>(a, grid, stream);
    case 4 * 4 + 2: return launch<2, 4>(a, grid, stream);
  }
  *handled = false;
  return FAIRY2I_OK;
}

}  // namespace fairy2i
