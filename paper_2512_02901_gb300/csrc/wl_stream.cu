// Persistent decode (B <= 2 tokens) kernel of the quantized widely-linear matmul on the
// 5th-generation tensor cores: the packed codes stream through shared memory, are decoded into
// tensor memory and multiplied there (tcgen05.mma with A in TMEM).
//
// Arithmetic (Eq. ifairy-dequant, Algorithm 1 with the W conj(x) term). Every code carries the
// signs sigma = sign(Re b + Im b), tau = sign(Re b - Im b) of its codeword b; with
// h = (s_re + i s_im)/2 the dequantized weight is h sigma + conj(h) tau. Per (stage t, matrix)
// a row needs P = sum_k sigma_k x_k and Q = sum_k tau_k x_k; then y += h P + conj(h) Q for U and
// h conj(P) + conj(h) conj(Q) for W (the conj(x) term of Eq. widely-linear).
//
// Tensor-core form. TMEM lane L = tm R + r holds row r of stage-matrix tm = 2 t + matrix
// (R = 64, 32, 16, 16 rows for T = 1..4); an MMA has M = 128 and accumulates in f32. The time
// of one MMA follows the bytes of A it reads from TMEM, not N, so A is kept small and x is
// spread over the N columns.
// * One token: kind::mxf4 (e2m1 x e2m1, unit ue8m0 scale factors), K = 64. A code word (16
//   codes) becomes four A registers of eight nibbles, +1 = 0x2 or -1 = 0xA, four sigma and four
//   tau each (one shift and one LOP3 per register), so one MMA covers two words. x is
//   X = rn(|x| S) < 2^26 (S a power of two per CTA) in thirteen base-4 digits d_l, held as the
//   e2m1 values +-d_l / 2 with the sign of x, in the first 52 of 64 columns (slot, re/im, limb):
//   the sigma slot has them at the sigma positions of K and zeros at the tau positions, the tau
//   slot the reverse. The sums of digits are exact in f32, and P = (2 / S) sum_l 4^l D_l.
// * Two tokens: kind::f8f6f4 (e4m3), K = 32, one MMA per word. A word becomes 32 A bytes
//   (sigma_2j, sigma_2j+1, tau_2j, tau_2j+1) for j = 0..7, each an e4m3 value affine in its bit
//   by one LOP3 per four bytes (a = alpha + 2 bit, sigma = (1 + alpha) - a), so P = C - D, D the
//   MMA result and C = sum_k (1 + alpha_k) x_k the same for every row. B holds x split exactly
//   into two e4m3 limbs (hi = e4m3(x S), lo = e4m3(64 (x S - hi)), S a power of two per CTA and
//   token) in the 16 columns (token, limb, sigma/tau slot, re/im). The e2m1 form of two tokens
//   would need 96 accumulator columns per set.
//
// Work. A job is one row block (R rows of every stage-matrix) of one linear of the group; the
// jobs are dealt round-robin to thread-block clusters of ks CTAs, and rank r of a cluster takes
// the 128-code chunks [r nch / ks, (r+1) nch / ks) of every job, so a CTA's K range (and its
// x-dependent operands: the B tiles, C and S) is the same for all its jobs and is built once per
// launch. A unit is one chunk of one job (4 KB of codes: one 512-byte block per 16-row tile of
// every stage-matrix); a stage of the shared-memory ring holds one job's units, which arrive as
// one bulk copy per tile (the chunks of a tile are adjacent in memory). The grid holds at most
// one wave of resident clusters, so every CTA loops over its jobs and the launch has no tail
// wave. Partial rows are summed in distributed shared memory in rank order (deterministic);
// rank 0 writes y.
//
// Programmatic dependent launch. Only x (and y) may belong to the previous kernel in the stream:
// the copies of the codes into the shared-memory ring and their decoding into tensor memory
// start before griddepcontrol.wait; the B tiles, and with them every MMA, come after it.
//
// Roles: warps 0-7 are two decoder sets of four (warp w reaches TMEM lanes 32 (w % 4) ..), set s
// decoding units q = s, s + 2, ... into its three A slots; warp 8 streams the codes; lane 0 of
// warp 9 + s (e2m1) or of warps 9 + 2 s + e (e4m3: words 4e .. 4e + 3) issues the MMAs of every
// unit of set s into its own accumulator of the job's buffer (two buffers, so a job's read-out
// overlaps the next job's MMAs); the last four warps load x, build the B tiles (and C) and S,
// then read out, combine and reduce every job's accumulators and write y.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_fp8.h>

#include <mutex>

#include "common.cuh"
#include "ptx.cuh"
#include "tc.cuh"

namespace fairy2i {

namespace sd {

constexpr int kSets = 2;                      // decoder sets of four warps
constexpr int kDecWarps = 4 * kSets;          // warps 0-7
constexpr int kCopyWarp = kDecWarps;          // 8
constexpr int kIssWarp0 = kCopyWarp + 1;      // warp kIssWarp0 + kIss s + e
constexpr int kEpiThreads = 128;
constexpr int kRingBytes = 112 * 1024;        // code ring: one job (nu units) per stage
constexpr int kMaxStages = 14;
constexpr int kUnitBytes = 4096;              // codes of one unit (8 tiles x 512 B)
constexpr int kMaxU = 12;                     // chunks per CTA
constexpr int kMaxCluster = 8;
constexpr int kMaxGroup = 4;
constexpr int kTmemCols = 512;
constexpr uint64_t kWaitNs = 1000000000ull;   // 1 s: a pipeline wait is microseconds
// Base-4 digits of x in the e2m1 form: 2^-26 of the largest |x| of a CTA's K slice (at most
// 2 kMaxU 128 = 3072 real values) bounds the error of every x entry, so the x error in l1 norm
// stays below 3072 2^-26 = 4.6e-5 of |x|_1, within the 1e-4 |x|_1 sum_t s_t bound per output
// for any input.
constexpr int kLimbs4 = 13;

// Operand form and layout. One token (NB = 1): e2m1 (kind::mxf4), two codes' signs per A byte,
// one MMA (K = 64) per two code words, x as kLimbs4 base-4 digits in the first 52 of 64 B
// columns (slot, part, limb); three issuing threads per set taking every third unit of the set,
// all six adding into one accumulator per job buffer (a thread blocks for about 150 cycles on
// every MMA it issues, so units overlap only across threads; the digit sums are integers, exact in
// f32, so the order of the threads' MMAs does not matter; the epilogue zeroes the accumulator
// after reading it), which leaves tensor memory for five A slots per set. Two
// tokens: e4m3 (kind::f8f6f4), one MMA (K = 32) per word, x as two e4m3 limbs in 16 B columns
// (token, limb, slot, part); two issuing threads per set (words 0-3, 4-7), each into its own
// accumulator. The e2m1 form of two tokens would need 96 accumulator columns per set.
template <int NB>
struct Layout {
  static constexpr bool kF4 = NB == 1;
  static constexpr int kSlots = kF4 ? 5 : 3;                // A slots per set (one unit each)
  static constexpr int kIss = kF4 ? 3 : 2;                  // MMA-issuing threads per set
  static constexpr int kIssThreads = kSets * kIss;
  static constexpr int kNumAcc = kF4 ? 1 : kSets * kIss;    // accumulators per job buffer
  static constexpr int kNUsed = kF4 ? 2 * 2 * kLimbs4 : 16; // B columns holding x
  static constexpr int kN = (kNUsed + 15) / 16 * 16;        // MMA N (the rest zero)
  static constexpr int kPart = 128 * NB;                    // floats of one partial (R NB 2)
  static constexpr int kAccStride = kF4 ? 64 : 16;          // TMEM columns per accumulator
  static constexpr int kColSlots = 2 * kNumAcc * kAccStride;   // accumulators [buffer][set][issuer]
  static constexpr int kSlotCols = kF4 ? 32 : 64;           // TMEM columns of one unit's A
  static constexpr int kColSF = kColSlots + kSets * kSlots * kSlotCols;   // scale factors (e2m1)
  static constexpr int kMmas = kF4 ? 4 : 8;                 // MMAs per unit
  // B tile of one MMA: kN rows x 32 bytes, + 16 B so that consecutive tiles start in different
  // shared-memory banks.
  static constexpr int kMmaB = kN * 32 + 16;
  static constexpr int kChunkB = kMmas * kMmaB;             // B tiles of one chunk
  static constexpr uint32_t kIdesc = kF4 ? idesc_mxf4_f32(128, kN) : idesc_e4m3_f32(128, kN);
  static constexpr int kEpiWarp0 = kIssWarp0 + kSets * kIss;   // four warps, every warp % 4
  static constexpr int kWarps = kEpiWarp0 + 4;
  static constexpr int kThreads = kWarps * 32;
  // Shared memory (bytes from the 1024-aligned base).
  static constexpr int kOffRing = 0;
  static constexpr int kOffB = kOffRing + kRingBytes;
  static constexpr int kOffRed = kOffB + kMaxU * kChunkB;
  static constexpr int kOffGather = kOffRed + 128 * 2 * 2 * 4;
  static constexpr int kOffOut = kOffGather + 2 * kMaxCluster * kPart * 4;
  static constexpr int kOffBar = kOffOut + kPart * 4;
  static constexpr int kNumBars = 2 * kMaxStages + 2 * kSets * kSlots + 2 + 2 + 1 + 2 + 2 + kIssThreads + 1;
  static constexpr int kOffMisc = kOffBar + kNumBars * 8;
  static constexpr int kSmemBytes = kOffMisc + 512 + 1024;   // + alignment slack
  static_assert(kColSF + (kF4 ? 64 : 0) <= kTmemCols, "TMEM columns");
  // One CTA per SM: it owns all TMEM columns (a second CTA on the SM would wait in its
  // allocation), and no two CTAs of a launch share an SM's tensor core.
  static_assert(kSmemBytes > 116 * 1024, "one CTA per SM");
  static_assert(kSmemBytes <= 227 * 1024, "shared memory per CTA");
};

struct Args {
  const uint32_t* codes[kMaxGroup];
  const float* scales[kMaxGroup];
  float* y[kMaxGroup];
  const __nv_bfloat16* x;
  unsigned int* status;
  int64_t B, in_features, ldx, n, m, out_features, ldy;
  int G;          // linears in the group
  int nch;        // 128-code chunks per row
  int row_tiles;  // ceil(n / 16)
  int rbs;        // row blocks per linear, ceil(n / R)
  int ks;         // CTAs per cluster
  int nclusters;  // clusters in the grid
  int x_vec;      // x rows 16-byte aligned with m % 8 == 0: vector loads allowed
  int x_bulk;     // and in_features even: the x slice is prefetched to L2 in one range
};

struct Misc {
  uint32_t tmem;
  int abort;
  unsigned int xmax[4][2];       // per epilogue warp and token: max |x| as float bits
  float scl[kMaxGroup][16];      // scales of the group: [linear][(stage, matrix, re/im)]
  float cpart[4][4];             // per epilogue warp: [token][part] partial C
};

// Bulk copy of `bytes` (a multiple of 16) from this CTA's shared memory to the shared memory of
// another CTA of the cluster, completing its bytes on an mbarrier there (cluster addresses).
__device__ __forceinline__ void bulk_copy_to_cluster(uint32_t dst, uint32_t src, uint32_t bytes,
                                                     uint32_t mbar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(dst), "r"(src), "r"(bytes), "r"(mbar)
      : "memory");
}
// Waits until the bulk copies this thread issued have read their sources.
__device__ __forceinline__ void bulk_commit_wait_read() {
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}

__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, volatile int* abort,
                                              unsigned int* status) {
  if (*abort) return false;
  if (mbar_wait_poll(bar, parity, kWaitNs)) return true;
  *abort = 1;
  latch_status(status, kStatusTimeout);
  return false;
}

// A register j (0..7) of a word: e4m3 bytes (sigma_2j, sigma_2j+1, tau_2j, tau_2j+1), each
// alpha_q + 2 bit with q the bit position used (2, 3, 2, 3, 6, 7, 6, 7 for j = 0..7; the word
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

// e2m1 form: the four A registers of a word. The word holds the sign bits of sigma in bits 0-15
// and of tau in bits 16-31, code i at bit 8 (i % 2) + i / 2 of its half. Register s keeps the
// bits 4 n + 3 - s of the word as the sign bits (4 n + 3) of nibbles n = 0..7 on the magnitude
// 1 (0x2): nibbles 0-3 are sigma and nibbles 4-7 tau of the codes at bits 4 n + 3 - s of the
// halves (0x2 = +1, 0xA = -1). One shift and one LOP3 per register.
__device__ __forceinline__ void decode_word4(uint32_t w, uint32_t* r) {
  r[0] = lop3_and_or(w, 0x88888888u, 0x22222222u);
  r[1] = lop3_and_or(w << 1, 0x88888888u, 0x22222222u);
  r[2] = lop3_and_or(w << 2, 0x88888888u, 0x22222222u);
  r[3] = lop3_and_or(w << 3, 0x88888888u, 0x22222222u);
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

// Eight bf16 values of part `part` of token b at complex index k (k % 8 == 0), zero outside
// the valid range of that part. Plain (coherent) loads: x may come from the previous kernel.
__device__ __forceinline__ uint4 load_x8(const Args& a, int b, int part, int64_t k) {
  const __nv_bfloat16* row = a.x + (int64_t)b * a.ldx + (int64_t)part * a.m;
  const int64_t lim = part ? a.in_features - a.m : a.m;
  if (a.x_vec && k + 8 <= lim) return *reinterpret_cast<const uint4*>(row + k);
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

// Job index i of this cluster -> (linear g, row block rb).
__device__ __forceinline__ void job_of(const Args& a, int cluster, int i, int& g, int& rb) {
  const int J = cluster + i * a.nclusters;
  g = J / a.rbs;
  rb = J - g * a.rbs;
}

template <int NB, int T>
__global__ void __launch_bounds__(Layout<NB>::kThreads, 1) wl_stream_kernel(const Args a) {
  using Lay = Layout<NB>;
  constexpr bool kF4 = Lay::kF4;
  constexpr int kSlots = Lay::kSlots, kIss = Lay::kIss, kNumAcc = Lay::kNumAcc;
  constexpr int kIssThreads = Lay::kIssThreads;
  static_assert(!kF4 || kSlots >= kIss, "an issuer never waits two phases ahead on a slot");
  constexpr int kEpiWarp0 = Lay::kEpiWarp0;
  constexpr int kColSlots = Lay::kColSlots, kSlotCols = Lay::kSlotCols;
  constexpr int kAccStride = Lay::kAccStride, kMmaB = Lay::kMmaB, kChunkB = Lay::kChunkB;
  constexpr int kOffRing = Lay::kOffRing, kOffB = Lay::kOffB, kOffRed = Lay::kOffRed;
  constexpr int kOffGather = Lay::kOffGather, kOffOut = Lay::kOffOut, kOffBar = Lay::kOffBar;
  constexpr int kOffMisc = Lay::kOffMisc, kNumBars = Lay::kNumBars;
  constexpr int TM = 2 * T;
  constexpr int R = (T == 1) ? 64 : (T == 2 ? 32 : 16);  // rows per row block
  constexpr int RT = R / 16;                              // 16-row code tiles per row block
  constexpr int NV = R * NB * 2;                          // outputs of a row block
  static_assert(TM * RT * 512 <= kUnitBytes, "unit size");
  constexpr int kPart = Lay::kPart;
  static_assert(NV <= kPart && NV <= 2 * kEpiThreads, "partial size");
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = align_smem_1024(smem_raw);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kOffBar);
  uint64_t* full = bars;                        // [stage] codes landed        (tx count)
  uint64_t* empty = full + kMaxStages;          // [stage] codes read          (4 warps x nu)
  uint64_t* sfull = empty + kMaxStages;         // [set][slot] A written       (4 warps)
  uint64_t* sfree = sfull + kSets * kSlots;     // [set][slot] its MMAs done   (e2m1: 1, e4m3: kIss commits)
  uint64_t* jfull = sfree + kSets * kSlots;     // [buffer] job accumulated    (every issuer)
  uint64_t* jfree = jfull + 2;                  // [buffer] job read out       (4 warps)
  uint64_t* bready = jfree + 2;                 // B tiles written             (1 arrival)
  uint64_t* gfull = bready + 1;                 // [buffer] rank 0: partials arrived
  uint64_t* gfree = gfull + 2;                  // [buffer] ranks > 0: rank 0 read the buffer
  uint64_t* fin = gfree + 2;                    // [issuer] abort path
  uint64_t* sfready = fin + kIssThreads;        // e2m1: scale factors written (4 warps)
  Misc* misc = reinterpret_cast<Misc*>(smem + kOffMisc);
  volatile int* abort_flag = &misc->abort;
  float* red = reinterpret_cast<float*>(smem + kOffRed);
  float* gather = reinterpret_cast<float*>(smem + kOffGather);          // [buf][rank][kPart]
  float* outp = reinterpret_cast<float*>(smem + kOffOut);               // partial sent to rank 0

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int ks = a.ks;
  const int rank = ks > 1 ? (int)cluster_ctarank() : 0;
  const int cluster = (int)(blockIdx.x / (unsigned)ks);
  const int c0 = (rank * a.nch) / ks;
  const int nu = ((rank + 1) * a.nch) / ks - c0;          // units per job (>= 1)
  const int njobs_all = a.G * a.rbs;
  const int njobs = cluster < njobs_all ? (njobs_all - 1 - cluster) / a.nclusters + 1 : 0;
  const int total = njobs * nu;                           // units of this CTA
  const int stage_bytes = nu * kUnitBytes;                // one job: [tile][unit][512 B]
  const int nstages = min(kMaxStages, kRingBytes / stage_bytes);

  // ---- prologue: barriers (the lanes of warp 1), TMEM (warp 0) ----
  if (warp == 1) {
    for (int i = lane; i < kNumBars; i += 32) {
      uint32_t cnt = 1;
      if (i >= kMaxStages && i < 2 * kMaxStages) cnt = 4 * nu;                         // empty
      else if (i >= 2 * kMaxStages && i < 2 * kMaxStages + kSets * kSlots) cnt = 4;    // sfull
      else if (i < 2 * kMaxStages + 2 * kSets * kSlots && i >= 2 * kMaxStages) cnt = kF4 ? 1 : kIss;
      else if (bars + i == jfull || bars + i == jfull + 1) cnt = kIssThreads;
      else if (bars + i == jfree || bars + i == jfree + 1) cnt = 4;
      else if (bars + i == sfready) cnt = 4;
      mbar_init(bars + i, cnt);
    }
    if (lane == 0) misc->abort = 0;
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&misc->tmem, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = misc->tmem;
  if (kF4 && warp < 4) {
    // Unit scale factors (ue8m0 127 = 1.0) for every row of A and B of every MMA; the issuing
    // threads wait for them on sfready (off the other roles' path).
    uint32_t ones[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) ones[i] = 0x7F7F7F7Fu;
    const uint32_t la = tmem + ((uint32_t)(warp * 32) << 16) + Lay::kColSF;
    tmem_st32(la, ones);
    tmem_st32(la + 32, ones);
    // the shared accumulators start at zero (every MMA adds)
#pragma unroll
    for (int i = 0; i < 32; ++i) ones[i] = 0u;
    const uint32_t lz = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll
    for (int c = 0; c < kColSlots; c += 32) tmem_st32(lz + c, ones);
    tmem_wait_st();
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(sfready);
  }
  if (ks > 1) cluster_arrive_relaxed();   // every rank's barriers initialised (waited before DSMEM use)
  pdl_launch_dependents();

  if (warp < kDecWarps) {
    // ---------------- decoder sets: one unit into one A slot at a time ----------------
    const int set = warp >> 2, quarter = warp & 3;
    const int L = quarter * 32 + lane;                       // TMEM lane of this thread
    const int tm = L / R, r = L % R;
    // this lane's 8 words of unit u inside a stage: tile tm RT + r / 16, row r % 16 (32 bytes)
    const uint32_t lane_off = (uint32_t)((tm * RT + r / 16) * nu * 512 + (r % 16) * 32);
    const uint32_t ring = smem_u32(smem + kOffRing);
    const uint32_t t_lane = tmem + ((uint32_t)(quarter * 32) << 16) + kColSlots;
    // unit q = set + kSets l: chunk u of job i, in ring stage st (its (i / nstages)-th use,
    // phase fph) and A slot sl of the set (its (l / kSlots)-th use, phase ph); no divisions
    int i = 0, u = set, st = 0, sl = 0;
    uint32_t fph = 0, ph = 0;
    auto next_job = [&]() {
      ++i;
      if (++st == nstages) {
        st = 0;
        fph ^= 1u;
      }
    };
    while (u >= nu) {
      u -= nu;
      next_job();
    }
    int l = 0;
    for (int q = set; q < total; q += kSets, ++l) {
      const int si = set * kSlots + sl;
      if (!__all_sync(0xffffffffu, mbar_test_wait(&full[st], fph) ||
                                       wait_or_abort(&full[st], fph, abort_flag, a.status)))
        break;
      const uint32_t src = ring + st * stage_bytes + lane_off + u * 512;
      const uint4 q0 = lds128(src), q1 = lds128(src + 16);
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);
      // Units past the first kSlots need MMAs, i.e. x: wait for the previous kernel first, so
      // that no bounded wait below counts its run time.
      if (l == kSlots) pdl_wait_primary();
      if (l >= kSlots) {   // the slot's previous unit has been multiplied
        if (!__all_sync(0xffffffffu, mbar_test_wait(&sfree[si], ph ^ 1u) ||
                                         wait_or_abort(&sfree[si], ph ^ 1u, abort_flag, a.status)))
          break;
        tc_fence_after();   // the stores below follow the MMAs that read the slot
      }
      const uint32_t a_col = t_lane + si * kSlotCols;
      uint32_t rr[32];
      if constexpr (kF4) {   // word w -> columns 4 w .. 4 w + 3
        decode_word4(q0.x, rr);
        decode_word4(q0.y, rr + 4);
        decode_word4(q0.z, rr + 8);
        decode_word4(q0.w, rr + 12);
        decode_word4(q1.x, rr + 16);
        decode_word4(q1.y, rr + 20);
        decode_word4(q1.z, rr + 24);
        decode_word4(q1.w, rr + 28);
        tmem_st32(a_col, rr);
      } else {               // word w -> columns 8 w .. 8 w + 7
        decode_word(q0.x, rr);
        decode_word(q0.y, rr + 8);
        decode_word(q0.z, rr + 16);
        decode_word(q0.w, rr + 24);
        tmem_st32(a_col, rr);
        decode_word(q1.x, rr);
        decode_word(q1.y, rr + 8);
        decode_word(q1.z, rr + 16);
        decode_word(q1.w, rr + 24);
        tmem_st32(a_col + 32, rr);
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sfull[si]);
      if (++sl == kSlots) {
        sl = 0;
        ph ^= 1u;
      }
      u += kSets;
      while (u >= nu) {
        u -= nu;
        next_job();
      }
    }
  } else if (warp == kCopyWarp) {
    // ---------------- code stream: one stage per job, one bulk copy per tile ----------------
    const int tmi = lane / RT, rt = lane % RT;
    const uint64_t pol = l2_evict_first_policy();   // the codes are read once per launch
    int issued = 0;
    for (int i = 0; i < njobs; ++i) {
      const int st = i % nstages;
      if (i == nstages) pdl_wait_primary();   // refills wait on MMAs, i.e. on x
      if (i >= nstages) {
        const bool ok = lane != 0 || wait_or_abort(&empty[st], ((i / nstages) - 1) & 1,
                                                   abort_flag, a.status);
        if (!__all_sync(0xffffffffu, ok)) break;
      }
      int g, rb;
      job_of(a, cluster, i, g, rb);
      int nrt = 0;   // existing 16-row tiles of the row block
#pragma unroll
      for (int k = 0; k < RT; ++k) nrt += (rb * RT + k < a.row_tiles) ? 1 : 0;
      if (lane == 0) mbar_arrive_expect_tx(&full[st], (uint32_t)(TM * nrt * nu * 512));
      __syncwarp();
      if (lane < TM * RT && rt < nrt) {
        const int64_t tile = (int64_t)tmi * a.row_tiles + rb * RT + rt;
        bulk_load_hint(smem + kOffRing + st * stage_bytes + lane * nu * 512,
                       a.codes[g] + (tile * a.nch + c0) * 128, (uint32_t)(nu * 512), &full[st],
                       pol);
      }
      issued = i + 1;
    }
    // Abort path: every issued copy lands before shared memory is released.
    if (lane == 0 && *abort_flag) {
      for (int i = (issued > nstages ? issued - nstages : 0); i < issued; ++i)
        (void)mbar_wait_timed(&full[i % nstages], (i / nstages) & 1, 1000000ull);
    }
  } else if (warp < kEpiWarp0) {
    // ------ MMA issuers: lane 0 of warp kIssWarp0 + kIss s + e issues, e2m1: the units
    // l = e, e + kIss, ... of set s into the set's accumulator of the job's buffer; e4m3: words
    // 4e .. 4e+3 of every unit of set s into its own accumulator ------
    const int ii = warp - kIssWarp0, set = ii / kIss, e = ii % kIss;
    if (lane == 0) {
      const uint32_t b_base = smem_u32(smem + kOffB);
      // the scale factors are stored long before the B tiles: waited off the critical path
      bool ok = !kF4 || wait_or_abort(sfready, 0, abort_flag, a.status);
      pdl_wait_primary();   // the B tiles are built from x after the previous kernel
      if (ok) ok = wait_or_abort(bready, 0, abort_flag, a.status);
      tc_fence_after();
      bool issued = false;
      int cur = -1;
      bool first = true;
      // Before touching job i's accumulator buffer, the read-out of job i - 2 must be done; a
      // job without a unit of this set still gets this issuer's arrival.
      auto enter_job = [&](int i) {
        if (i >= 2 && ok) ok = wait_or_abort(&jfree[i & 1], ((i >> 1) - 1) & 1, abort_flag, a.status);
      };
      // Unit q = set + kSets l of the CTA is chunk u of job i, in slot sl = l % kSlots of the
      // set for the (l / kSlots)-th time (phase ph); this thread takes l = l0, l0 + lstep, ...
      // (e2m1: l0 = e, lstep = kIss; e4m3: every unit). Advanced without divisions in the loop,
      // since this thread's loop overhead adds to every unit.
      constexpr int lstep = kF4 ? kIss : 1;
      const int l0 = kF4 ? e : 0;
      int i = 0, u = set + kSets * l0, sl = l0 % kSlots;
      uint32_t ph = (uint32_t)(l0 / kSlots) & 1u;
      while (u >= nu) {
        u -= nu;
        ++i;
      }
      const uint64_t desc0 = smem_desc(b_base, 128, 256);   // + (byte offset >> 4) per tile
      for (int q = set + kSets * l0; ok && q < total; q += kSets * lstep) {
        if (i != cur) {
          if (cur >= 0) mma_commit(&jfull[cur & 1]);
          for (int i2 = cur + 1; ok && i2 < i; ++i2) {   // jobs without a unit of this thread
            enter_job(i2);
            if (ok) mbar_arrive(&jfull[i2 & 1]);
          }
          enter_job(i);
          if (!ok) break;
          tc_fence_after();
          cur = i;
          first = true;
        }
        const int si = set * kSlots + sl;
        ok = mbar_test_wait(&sfull[si], ph) || wait_or_abort(&sfull[si], ph, abort_flag, a.status);
        if (!ok) break;
        tc_fence_after();
        const uint32_t a_slot = tmem + kColSlots + si * kSlotCols;
        const uint64_t bd = desc0 + (uint64_t)((u * kChunkB) >> 4);
        if constexpr (kF4) {   // MMA j: words 2 j, 2 j + 1 (A columns 8 j ..); every MMA adds
          const uint32_t d_tmem = tmem + (cur & 1) * kAccStride;
#pragma unroll
          for (int j = 0; j < 4; ++j)
            mma_mxf4_ts(d_tmem, a_slot + j * 8, bd + (uint64_t)((j * kMmaB) >> 4), Lay::kIdesc,
                        tmem + Lay::kColSF, tmem + Lay::kColSF + 16, 1u);
        } else {               // MMA w: word w (A columns 8 w ..)
          const uint32_t d_tmem = tmem + ((cur & 1) * kNumAcc + ii) * kAccStride;
#pragma unroll
          for (int w4 = 0; w4 < 4; ++w4) {
            const int w = e * 4 + w4;
            mma_e4m3_ts(d_tmem, a_slot + w * 8, bd + (uint64_t)((w * kMmaB) >> 4), Lay::kIdesc,
                        (first && w4 == 0) ? 0u : 1u);
          }
        }
        first = false;
        issued = true;
        mma_commit(&sfree[si]);
        sl += lstep;   // lstep < kSlots: at most one wrap
        if (sl >= kSlots) {
          sl -= kSlots;
          ph ^= 1u;
        }
        u += kSets * lstep;
        while (u >= nu) {
          u -= nu;
          ++i;
        }
      }
      if (ok) {
        if (cur >= 0) mma_commit(&jfull[cur & 1]);
        for (int i2 = cur + 1; ok && i2 < njobs; ++i2) {
          enter_job(i2);
          if (ok) mbar_arrive(&jfull[i2 & 1]);
        }
      }
      // Abort path: the MMAs this thread issued finish before TMEM is released.
      if (issued && *abort_flag) {
        mma_commit(&fin[ii]);   // ii < kIssThreads
        (void)mbar_wait_timed(&fin[ii], 0, kWaitNs);
      }
    }
    __syncwarp();
  } else {
    // ---------------- x -> B tiles, C, S; then the read-out of every job ----------------
    const int et = tid - kEpiWarp0 * 32;        // 0 .. 127
    const int ew = warp - kEpiWarp0;            // 0 .. 3
    const int quarter = warp & 3;
    const int L = quarter * 32 + lane;
    const int64_t kbeg = (int64_t)c0 * 128;
    // Before the wait: zero the B tiles (rows of unused tokens stay zero) and warm L2 with the
    // x slice.
    if constexpr (!kF4) {
      for (int o = et; o < nu * kChunkB / 16; o += kEpiThreads)
        *reinterpret_cast<uint4*>(smem + kOffB + o * 16) = make_uint4(0, 0, 0, 0);
    } else {   // the rows past the digits, 16 bytes (row, half) at a time
      constexpr int kSpare = (Lay::kN - Lay::kNUsed) * 2;
      for (int o = et; o < nu * Lay::kMmas * kSpare; o += kEpiThreads) {
        const int tile = o / kSpare, rest = o % kSpare, n = Lay::kNUsed + (rest >> 1);
        *reinterpret_cast<uint4*>(smem + kOffB + tile * kMmaB + (n >> 3) * 256 + (rest & 1) * 128 +
                                  (n & 7) * 16) = make_uint4(0, 0, 0, 0);
      }
    }
    // the scales, like the codes, are not written by the previous kernel
    // (stored into shared memory after the B tiles: the load's latency stays off the path to x)
    const float scl_v = et < a.G * TM * 2 ? __ldg(a.scales[et / (TM * 2)] + et % (TM * 2)) : 0.f;
    if (a.x_bulk && et < 2 * NB && et / 2 < a.B) {
      const int b = et >> 1, p = et & 1;
      const int64_t lim = p ? a.in_features - a.m : a.m;
      const int64_t k1 = min((int64_t)(c0 + nu) * 128, lim);
      if (k1 > kbeg)
        prefetch_l2_bulk(a.x + (int64_t)b * a.ldx + (int64_t)p * a.m + kbeg,
                         (uint32_t)((k1 - kbeg) * 2));
    }
    pdl_wait_primary();               // x may be written by the previous kernel
    // e4m3: x S in two limbs, P = C - D; e2m1: X = |x| S in base-4 digits
    float S[2] = {1.f, 1.f}, invS[2] = {1.f, 1.f}, C[4] = {0.f, 0.f, 0.f, 0.f};
    if constexpr (kF4) {
      // Items it = (8 u + w) 2 + p of the slice: the 16 values x_p[kbeg + 128 u + 16 w + i],
      // i = 0..15, of code word w of chunk u (two items per thread at most).
      static_assert(16 * kMaxU <= 2 * kEpiThreads, "x items per thread");
      uint4 xv[2][2];
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int it = et + j * kEpiThreads;
        xv[j][0] = xv[j][1] = make_uint4(0, 0, 0, 0);
        if (it < nu * 16) {
          const int64_t k = kbeg + 128 * (it >> 4) + 16 * ((it >> 1) & 7);
          xv[j][0] = load_x8(a, 0, it & 1, k);
          xv[j][1] = load_x8(a, 0, it & 1, k + 8);
        }
      }
      unsigned int mx = 0u;   // max |x| (non-negative float bits order like unsigned integers)
#pragma unroll
      for (int j = 0; j < 2; ++j)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const uint32_t ev[4] = {xv[j][h].x, xv[j][h].y, xv[j][h].z, xv[j][h].w};
#pragma unroll
          for (int i = 0; i < 4; ++i) mx = max(mx, max((ev[i] << 17) >> 1, ev[i] & 0x7fff0000u));
        }
      mx = __reduce_max_sync(0xffffffffu, mx);
      if (lane == 0) misc->xmax[ew][0] = mx;
      named_bar_sync(1, kEpiThreads);
      const unsigned int xm = max(max(misc->xmax[0][0], misc->xmax[1][0]),
                                  max(misc->xmax[2][0], misc->xmax[3][0]));
      // S = 2^(26 - E) for 2^(E-1) <= max|x| < 2^E: every X = rn(|x| S) < 2^26 is kLimbs4
      // base-4 digits, and P = (2 / S) sum_l 4^l D_l with D_l the MMA column of digit l (e2m1
      // holds digit d as d / 2).
      const int se = min(254, max(1, 127 + 2 * kLimbs4 + 126 - (int)(xm >> 23)));
      S[0] = __uint_as_float((uint32_t)se << 23);
      invS[0] = 2.f / S[0];
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int it = et + j * kEpiThreads;
        if (it < nu * 16) {
          const int u = it >> 4, w = (it >> 1) & 7, p = it & 1;
          // register i of the item: codes 2 i (low half) and 2 i + 1 (high half)
          const uint32_t ev[8] = {xv[j][0].x, xv[j][0].y, xv[j][0].z, xv[j][0].w,
                                  xv[j][1].x, xv[j][1].y, xv[j][1].z, xv[j][1].w};
          // Row (slot, p, l) of the MMA tile of words 2 (w / 2), + 1, half w % 2: A register s
          // of the word pairs nibble n (n < 4) with sigma, nibble n + 4 with tau of the code at
          // bit q = 4 n + 3 - s of a half (code 2 q, or 2 (q - 8) + 1 for q >= 8). The sigma
          // slot holds digit l of x of that code in nibble n of word s, the tau slot in nibble
          // n + 4. The codes of words s = 0, 1 (group A) and s = 2, 3 (group B), nibble n of
          // word s at position 4 (s % 2) + n: X = rn(|x| S) of the eight values, transposed as an
          // 8 x 8 nibble matrix, gives in word j the nibble j (digits 2 j, 2 j + 1) of every
          // value, so digit l of all eight values is one shift and one LOP3.
          constexpr int kOrdA[8] = {6, 14, 7, 15, 4, 12, 5, 13};
          constexpr int kOrdB[8] = {2, 10, 3, 11, 0, 8, 1, 9};
          uint32_t XA[8], XB[8], sgA = 0u, sgB = 0u;
#pragma unroll
          for (int n = 0; n < 8; ++n) {
            const uint32_t va = ev[kOrdA[n] >> 1], vb = ev[kOrdB[n] >> 1];
            const float fa = (kOrdA[n] & 1) ? bf_hi(va) : bf_lo(va);
            const float fb = (kOrdB[n] & 1) ? bf_hi(vb) : bf_lo(vb);
            XA[n] = __float2uint_rn(fabsf(fa) * S[0]);
            XB[n] = __float2uint_rn(fabsf(fb) * S[0]);
            sgA |= (__float_as_uint(fa) >> 31) << (4 * n + 3);
            sgB |= (__float_as_uint(fb) >> 31) << (4 * n + 3);
          }
          transpose_nibbles(XA);
          transpose_nibbles(XB);
          unsigned char* tile = smem + kOffB + u * kChunkB + (w >> 1) * kMmaB + (w & 1) * 128;
#pragma unroll
          for (int l = 0; l < kLimbs4; ++l) {
            const uint32_t wa = lop3_and_or(XA[l >> 1] >> (2 * (l & 1)), 0x33333333u, sgA);
            const uint32_t wb = lop3_and_or(XB[l >> 1] >> (2 * (l & 1)), 0x33333333u, sgB);
            const uint32_t ws[4] = {wa & 0xffffu, wa >> 16, wb & 0xffffu, wb >> 16};
            const int ns = p * kLimbs4 + l, nt = (2 + p) * kLimbs4 + l;
            *reinterpret_cast<uint4*>(tile + (ns >> 3) * 256 + (ns & 7) * 16) =
                make_uint4(ws[0], ws[1], ws[2], ws[3]);
            *reinterpret_cast<uint4*>(tile + (nt >> 3) * 256 + (nt & 7) * 16) =
                make_uint4(wa << 16, wa & 0xffff0000u, wb << 16, wb & 0xffff0000u);
          }
        }
      }
      if (et < a.G * TM * 2) misc->scl[et / (TM * 2)][et % (TM * 2)] = scl_v;
      fence_proxy_async_smem();   // generic-proxy writes of B visible to the tensor cores
      named_bar_sync(1, kEpiThreads);
      if (et == 0) mbar_arrive(bready);
    } else {
      // This thread's groups: for token b and part p, the 8-value groups v = et + 128 jv of the
      // slice (v < 16 nu), values x_p[8 v .. 8 v + 7].
      constexpr int kJv = 2;                      // 16 kMaxU / 128 groups per (b, p) and thread
      static_assert(16 * kMaxU <= kJv * kEpiThreads, "x groups per thread");
      uint4 xv[NB][2][kJv];
#pragma unroll
      for (int b = 0; b < NB; ++b)
#pragma unroll
        for (int p = 0; p < 2; ++p)
#pragma unroll
          for (int jv = 0; jv < kJv; ++jv) {
            const int v = et + jv * kEpiThreads;
            xv[b][p][jv] = (v < nu * 16 && b < a.B) ? load_x8(a, b, p, kbeg + v * 8)
                                                    : make_uint4(0, 0, 0, 0);
          }
      // max |x| per token (non-negative float bits order like unsigned integers)
#pragma unroll
      for (int b = 0; b < NB; ++b) {
        unsigned int mx = 0u;
#pragma unroll
        for (int p = 0; p < 2; ++p)
#pragma unroll
          for (int jv = 0; jv < kJv; ++jv) {
            const uint32_t ev[4] = {xv[b][p][jv].x, xv[b][p][jv].y, xv[b][p][jv].z, xv[b][p][jv].w};
#pragma unroll
            for (int i = 0; i < 4; ++i) mx = max(mx, max((ev[i] << 17) >> 1, ev[i] & 0x7fff0000u));
          }
        mx = __reduce_max_sync(0xffffffffu, mx);
        if (lane == 0) misc->xmax[ew][b] = mx;
      }
      named_bar_sync(1, kEpiThreads);
#pragma unroll
      for (int b = 0; b < NB; ++b) {
        const unsigned int xm = max(max(misc->xmax[0][b], misc->xmax[1][b]),
                                    max(misc->xmax[2][b], misc->xmax[3][b]));
        pow2_scale(__uint_as_float(xm), S[b], invS[b]);
      }
      // B tiles and C. Group v = 16 u + 2 w + hh of token b, part p: the values x_p[k], k = 128 u +
      // 16 w + 8 hh .. + 7, become the 16-byte halves hh of the four rows (limb, slot, p) of token b
      // in the tile of word w of chunk u: register j' (codes 2j, 2j + 1, j = 4 hh + j') holds the
      // limb bytes of x[2j], x[2j + 1] in its sigma half (bytes 0-1) or tau half (bytes 2-3).
      float cacc[2][2] = {{0.f, 0.f}, {0.f, 0.f}};
#pragma unroll
      for (int b = 0; b < NB; ++b)
#pragma unroll
        for (int p = 0; p < 2; ++p)
#pragma unroll
          for (int jv = 0; jv < kJv; ++jv) {
            const int v = et + jv * kEpiThreads;
            if (v < nu * 16) {
              const int u = v >> 4, w = (v >> 1) & 7, hh = v & 1;
              const uint32_t ev[4] = {xv[b][p][jv].x, xv[b][p][jv].y, xv[b][p][jv].z,
                                      xv[b][p][jv].w};
              uint32_t hp[4], lp[4];   // limb byte pairs (x[2j], x[2j+1]) of register j'
              float cs = 0.f;
#pragma unroll
              for (int jj = 0; jj < 4; ++jj) {
                const float f0 = bf_lo(ev[jj]), f1 = bf_hi(ev[jj]);
                const float v0 = f0 * S[b], v1 = f1 * S[b];
                hp[jj] = e4m3x2(v0, v1) & 0xffffu;
                const float2 hf = e4m3x2_to_float2(hp[jj]);
                lp[jj] = e4m3x2(64.f * (v0 - hf.x), 64.f * (v1 - hf.y)) & 0xffffu;
                // 1 + alpha of codes 2j, 2j+1: 5, 3, 5, 3 (first half of a word), 1, 0, 1, 0
                const float wgt = hh ? ((jj & 1) ? 0.f : 1.f) : ((jj & 1) ? 3.f : 5.f);
                cs = fmaf(wgt, f0 + f1, cs);
              }
              cacc[b][p] += cs;
              unsigned char* tile = smem + kOffB + u * kChunkB + w * kMmaB;
#pragma unroll
              for (int limb = 0; limb < 2; ++limb) {
                const uint32_t* src = limb ? lp : hp;
#pragma unroll
                for (int slot = 0; slot < 2; ++slot) {
                  const int nrow = ((b * 2 + limb) * 2 + slot) * 2 + p;
                  const int sh = slot ? 16 : 0;
                  *reinterpret_cast<uint4*>(tile + (nrow >> 3) * 256 + hh * 128 + (nrow & 7) * 16) =
                      make_uint4(src[0] << sh, src[1] << sh, src[2] << sh, src[3] << sh);
                }
              }
            }
          }
      if (et < a.G * TM * 2) misc->scl[et / (TM * 2)][et % (TM * 2)] = scl_v;
      fence_proxy_async_smem();   // generic-proxy writes of B visible to the tensor cores
      named_bar_sync(1, kEpiThreads);
      if (et == 0) mbar_arrive(bready);
#pragma unroll
      for (int b = 0; b < 2; ++b)
#pragma unroll
        for (int p = 0; p < 2; ++p) {
          float v = cacc[b][p];
#pragma unroll
          for (int h = 16; h >= 1; h >>= 1) v += __shfl_xor_sync(0xffffffffu, v, h);
          if (lane == 0) misc->cpart[ew][b * 2 + p] = v;
        }
      named_bar_sync(1, kEpiThreads);
#pragma unroll
      for (int j = 0; j < 4; ++j)
        C[j] = (misc->cpart[0][j] + misc->cpart[1][j]) + (misc->cpart[2][j] + misc->cpart[3][j]);

    }

    // ---- per job: read out, combine with the scales, sum the stage-matrices, reduce ----
    if (ks > 1) cluster_wait();   // every rank's barriers are initialised
    const int tmL = L / R;
    for (int i = 0; i < njobs; ++i) {
      const int buf = i & 1;
      int g, rb;
      job_of(a, cluster, i, g, rb);
      float d[16];   // e4m3: columns (token, limb, slot, part)
#pragma unroll
      for (int k = 0; k < 16; ++k) d[k] = 0.f;
      float d4[4] = {0.f, 0.f, 0.f, 0.f};   // e2m1: sum_l 4^l D_l of (slot, part)
      const bool got = __all_sync(0xffffffffu,
                                  wait_or_abort(&jfull[buf], (i >> 1) & 1, abort_flag, a.status));
      tc_fence_after();
      // sets with at least one unit in job i
      auto has = [&](int s) { return nu >= kSets || ((s - i * nu) % kSets + kSets) % kSets < nu; };
      const uint32_t acc0 = tmem + ((uint32_t)(quarter * 32) << 16) + buf * kNumAcc * kAccStride;
      if (got) {
        if constexpr (kF4) {   // one accumulator per buffer: 64 columns
#pragma unroll
          for (int c16 = 0; c16 < Lay::kN / 16; ++c16) {
            float v[16];
            tmem_ld16(acc0 + c16 * 16, v);
            tmem_wait_ld();
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              const int col = c16 * 16 + k;   // (slot 2 + part) kLimbs4 + limb
              if (col < Lay::kNUsed)
                d4[col / kLimbs4] = fmaf(v[k], (float)(1u << (2 * (col % kLimbs4))),
                                         d4[col / kLimbs4]);
            }
          }
        } else {
#pragma unroll
          for (int s = 0; s < kSets; ++s) {
            if (has(s)) {
              float v0[16], v1[16];
              const uint32_t acc = acc0 + s * kIss * kAccStride;
              tmem_ld16(acc, v0);
              tmem_ld16(acc + kAccStride, v1);
              tmem_wait_ld();
#pragma unroll
              for (int k = 0; k < 16; ++k) d[k] += v0[k] + v1[k];
            }
          }
        }
      }
      if constexpr (kF4) {   // zero the accumulator of this buffer for job i + 2
        if (got) {
#pragma unroll
          for (int c = 0; c < kAccStride; c += 16) tmem_zero16(acc0 + c);
          tmem_wait_st();
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&jfree[buf]);
      if (L < TM * R) {
        const int t = tmL >> 1;
        const bool mat = tmL & 1;
        const float hr = 0.5f * misc->scl[g][(t * 2 + mat) * 2 + 0];
        const float hi = 0.5f * misc->scl[g][(t * 2 + mat) * 2 + 1];
        if constexpr (kF4) {
          const float is = invS[0];
          const float pre = d4[0] * is, qre = d4[2] * is;
          float pim = d4[1] * is, qim = d4[3] * is;
          if (mat) {   // W multiplies conj(x): conjugate P and Q
            pim = -pim;
            qim = -qim;
          }
          red[L * 2 + 0] = hr * pre - hi * pim + hr * qre + hi * qim;
          red[L * 2 + 1] = hr * pim + hi * pre + hr * qim - hi * qre;
        } else {
#pragma unroll
        for (int b = 0; b < NB; ++b) {
          const float cre = C[b * 2 + 0], cim = C[b * 2 + 1];
          const float is = invS[b];
          // column (token, limb, slot, part) = ((b 2 + limb) 2 + slot) 2 + part
          const int c = b * 8;
          const float pre = cre - (d[c + 0] + 0.015625f * d[c + 4]) * is;
          float pim = cim - (d[c + 1] + 0.015625f * d[c + 5]) * is;
          const float qre = cre - (d[c + 2] + 0.015625f * d[c + 6]) * is;
          float qim = cim - (d[c + 3] + 0.015625f * d[c + 7]) * is;
          if (mat) {   // W multiplies conj(x): conjugate P and Q
            pim = -pim;
            qim = -qim;
          }
          red[(L * NB + b) * 2 + 0] = hr * pre - hi * pim + hr * qre + hi * qim;
          red[(L * NB + b) * 2 + 1] = hr * pim + hi * pre + hr * qim - hi * qre;
        }
        }
      }
      named_bar_sync(1, kEpiThreads);
      // Sum over the stage-matrices: value idx = (row rr, token b, re/im).
      float vals[2];
#pragma unroll
      for (int it = 0; it < 2; ++it) {
        const int idx = et + it * kEpiThreads;
        float sum = 0.f;
        if (idx < NV) {
          const int rr = idx / (NB * 2), rest = idx % (NB * 2);
#pragma unroll
          for (int m2 = 0; m2 < TM; ++m2) sum += red[(m2 * R + rr) * NB * 2 + rest];
        }
        vals[it] = sum;
      }
      named_bar_sync(1, kEpiThreads);   // red is free for the next job
      bool write = rank == 0;
      if (ks > 1) {
        if (rank != 0) {
          // the buffer of job i - 2 in rank 0 has been read
          const bool fr = i < 2 || __all_sync(0xffffffffu, wait_or_abort(&gfree[buf], ((i >> 1) - 1) & 1,
                                                                        abort_flag, a.status));
          // Stage the partial, then one bulk copy into rank 0's gather slot, completing on rank 0's
          // barrier (also after an abort, so that rank 0 never waits for the full second).
          const bool ok2 = fr && !*abort_flag;
#pragma unroll
          for (int it = 0; it < 2; ++it) {
            const int idx = et + it * kEpiThreads;
            if (idx < NV) outp[idx] = ok2 ? vals[it] : 0.f;
          }
          fence_proxy_async_smem();
          named_bar_sync(1, kEpiThreads);
          if (et == 0) {
            const uint32_t g0 =
                smem_u32(gather) + (uint32_t)((buf * kMaxCluster + rank) * kPart) * 4;
            bulk_copy_to_cluster(mapa_shared(g0, 0), smem_u32(outp), (uint32_t)(NV * 4),
                                 mapa_shared(smem_u32(&gfull[buf]), 0));
            bulk_commit_wait_read();   // outp may be written again by the next job
          }
        } else {
          // Waited even after an abort: every rank sends its partial once per job, and rank 0
          // stays alive until those copies have landed.
          if (et == 0) mbar_arrive_expect_tx(&gfull[buf], (uint32_t)((ks - 1) * NV * 4));
          const bool got2 = __all_sync(0xffffffffu,
                                       mbar_wait_cluster_poll(&gfull[buf], (i >> 1) & 1, kWaitNs)) &&
                            !*abort_flag;
          if (!got2) {
            if (!*abort_flag) {
              *abort_flag = 1;
              latch_status(a.status, kStatusTimeout);
            }
            write = false;
          } else {
#pragma unroll
            for (int it = 0; it < 2; ++it) {
              const int idx = et + it * kEpiThreads;
              if (idx < NV)
                for (int r2 = 1; r2 < ks; ++r2) vals[it] += gather[(buf * kMaxCluster + r2) * kPart + idx];
            }
          }
          named_bar_sync(1, kEpiThreads);   // every read of gather[buf] is done
          // Rank r waits for this release only before job i + 2; the last two jobs send none, so
          // no remote access ever reaches a CTA that has passed its last wait.
          if (et < ks - 1 && i + 2 < njobs)
            mbar_arrive_remote(mapa_shared(smem_u32(&gfree[buf]), et + 1));
        }
      }
      if (write && !*abort_flag) {
#pragma unroll
        for (int it = 0; it < 2; ++it) {
          const int idx = et + it * kEpiThreads;
          if (idx < NV) {
            const int rr = idx / (NB * 2), b = (idx >> 1) % NB, comp = idx & 1;
            const int64_t jr = (int64_t)rb * R + rr;
            if (b < a.B && jr < a.n) {
              float* yb = a.y[g] + (int64_t)b * a.ldy;
              if (comp == 0) yb[jr] = vals[it];
              else if (a.n + jr < a.out_features) yb[a.n + jr] = vals[it];
            }
          }
        }
      }
    }
  }

  // Teardown. The first cluster barrier was waited by the epilogue warps; every other thread
  // waits it here. No second cluster barrier is needed: every remote access targets a CTA that
  // waits for it (rank 0 for the partials of every job, rank r > 0 for the release of a gather
  // buffer it writes again).
  if (ks > 1 && warp < kEpiWarp0) cluster_wait();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0) tmem_dealloc(tmem, kTmemCols);
}

template <int NB, int T>
fairy2i_status launch(const Args& a, int64_t grid, cudaStream_t stream) {
  auto kern = wl_stream_kernel<NB, T>;
  static std::atomic<uint64_t> smem_set{0};
  if (!smem_attr_once(kern, Layout<NB>::kSmemBytes, smem_set)) return FAIRY2I_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(Layout<NB>::kThreads);
  cfg.dynamicSmemBytes = Layout<NB>::kSmemBytes;
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

// Clusters of `ks` CTAs that can be resident at once on the device (0 if none).
template <int NB, int T>
int max_clusters(int ks) {
  auto kern = wl_stream_kernel<NB, T>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           Layout<NB>::kSmemBytes) != cudaSuccess)
    return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(ks * 256));
  cfg.blockDim = dim3(Layout<NB>::kThreads);
  cfg.dynamicSmemBytes = Layout<NB>::kSmemBytes;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)ks;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
    (void)cudaGetLastError();
    return 0;
  }
  return n;
}

}  // namespace sd

namespace {
std::mutex g_sd_mu;
int g_sd_clusters[64][4][8][2];   // [device][ks index][T][NB] resident clusters, -1 = unknown
bool g_sd_init[64];
}  // namespace

static int sd_resident_clusters(int dev, int ks_idx, int T, int NB) {
  std::lock_guard<std::mutex> lock(g_sd_mu);
  if (!g_sd_init[dev]) {
    for (int i = 0; i < 4; ++i)
      for (int t = 0; t < 8; ++t)
        for (int b = 0; b < 2; ++b) g_sd_clusters[dev][i][t][b] = -1;
    g_sd_init[dev] = true;
  }
  int& v = g_sd_clusters[dev][ks_idx][T - 1][NB - 1];
  if (v < 0) {
    const int ks = 1 << ks_idx;
    int r = 0;
    switch (T * 4 + NB) {
      case 1 * 4 + 1: r = sd::max_clusters<1, 1>(ks); break;
      case 1 * 4 + 2: r = sd::max_clusters<2, 1>(ks); break;
      case 2 * 4 + 1: r = sd::max_clusters<1, 2>(ks); break;
      case 2 * 4 + 2: r = sd::max_clusters<2, 2>(ks); break;
      case 3 * 4 + 1: r = sd::max_clusters<1, 3>(ks); break;
      case 3 * 4 + 2: r = sd::max_clusters<2, 3>(ks); break;
      case 4 * 4 + 1: r = sd::max_clusters<1, 4>(ks); break;
      case 4 * 4 + 2: r = sd::max_clusters<2, 4>(ks); break;
    }
    v = r;
  }
  return v;
}

// Cluster size and cluster count for `jobs` row blocks of `nch` chunks: ks in {1, 2, 4, 8} with
// at least one and at most kMaxU chunks per CTA, one wave of resident clusters of at most one CTA
// per SM, minimising the estimated time jobs-per-cluster x (chunks per CTA + a per-job cost of
// about a quarter chunk), then the fewest clusters that keep that busiest-cluster load.
struct SdPlan {
  int ks = 0, nclusters = 0;
};
static SdPlan sd_plan(int dev, int64_t jobs, int64_t nch, int T, int NB) {
  SdPlan best;
  int64_t best_cost = -1;
  int sms = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
    return best;
  for (int ki = 0; ki < 4; ++ki) {
    const int ks = 1 << ki;
    if (nch < ks || (nch + ks - 1) / ks > sd::kMaxU) continue;
    // one CTA per SM (the kernel's shared memory allows no second one)
    const int resident = std::min(sd_resident_clusters(dev, ki, T, NB), sms / ks);
    if (resident < 1) continue;
    const int64_t per = (jobs + resident - 1) / resident;     // jobs of the busiest cluster
    // the fewest clusters with that load: the SMs left free start the next kernel early
    const int64_t nclusters = (jobs + per - 1) / per;
    const int64_t cost = per * (4 * ((nch + ks - 1) / ks) + 1);   // a job's epilogue ~ 1/4 chunk
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best.ks = ks;
      best.nclusters = (int)nclusters;
    }
  }
  return best;
}

// `count` linears of the same shape sharing x. Handles B <= 2 bf16 tokens, T <= 4 and rows of at
// most 8 kMaxU chunks; anything else is left to the other kernels (*handled = false).
fairy2i_status launch_wl_stream_group(const void* x, fairy2i_dtype xdt, int64_t B,
                                      int64_t in_features, int64_t ldx, int count,
                                      const uint32_t* const* codes, const float* const* scales,
                                      int64_t n, int64_t m, int64_t out_features, int64_t wpr,
                                      int T, float* const* y, int64_t ldy, cudaStream_t stream,
                                      bool* handled) {
  using namespace sd;
  *handled = false;
  if (xdt != FAIRY2I_BF16 || B < 1 || B > 2 || T > 4 || count < 1 || count > kMaxGroup)
    return FAIRY2I_OK;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return FAIRY2I_ERR_CUDA;
  const int NB = (int)B;
  const int R = T == 1 ? 64 : (T == 2 ? 32 : 16);
  const int64_t rbs = (n + R - 1) / R;
  const int64_t nch = wpr / 8;
  const int64_t jobs = rbs * count;
  if (jobs > (int64_t(1) << 30) || nch > (int64_t(1) << 20)) return FAIRY2I_OK;
  const SdPlan plan = sd_plan(dev, jobs, nch, T, NB);
  if (plan.ks < 1) return FAIRY2I_OK;
  Args a;
  for (int g = 0; g < kMaxGroup; ++g) {
    a.codes[g] = codes[g < count ? g : 0];
    a.scales[g] = scales[g < count ? g : 0];
    a.y[g] = y[g < count ? g : 0];
  }
  a.x = reinterpret_cast<const __nv_bfloat16*>(x);
  a.status = device_status_word();
  a.B = B; a.in_features = in_features; a.ldx = ldx; a.n = n; a.m = m;
  a.out_features = out_features; a.ldy = ldy;
  a.G = count; a.nch = (int)nch; a.row_tiles = (int)((n + 15) / 16); a.rbs = (int)rbs;
  a.ks = plan.ks; a.nclusters = plan.nclusters;
  a.x_vec = (reinterpret_cast<uintptr_t>(x) % 16 == 0) && (ldx % 8 == 0) && (m % 8 == 0);
  a.x_bulk = a.x_vec && (in_features % 2 == 0);
  const int64_t grid = (int64_t)plan.nclusters * plan.ks;
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
