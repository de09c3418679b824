// Chained one-token decode of the quantized widely-linear matmul on the 5th-generation tensor
// cores: a sequence of calls (the linears of a decoder, in data-flow order) in one persistent
// launch. Call c reads its input only after every output of call c - 1 has been written, so a
// call may consume what the previous one produced; the packed codes, which do not depend on the
// data, stream through shared memory and are decoded into tensor memory ahead of time, across
// call boundaries.
//
// Arithmetic (Eq. ifairy-dequant, Algorithm 1 with the W conj(x) term). Every code carries the
// signs sigma = sign(Re b + Im b), tau = sign(Re b - Im b) of its codeword b, and with
// h = (s_re + i s_im)/2 the dequantized weight is h sigma + conj(h) tau. Per (stage t, matrix) a
// row needs P = sum_k sigma_k x_k and Q = sum_k tau_k x_k; then y += h P + conj(h) Q for U and
// h conj(P) + conj(h) conj(Q) for W (the conj(x) term of Eq. widely-linear).
//
// Tensor-core form: tcgen05.mma.kind::mxf4.block_scale (e2m1 x e2m1, f32 accumulate, unit ue8m0
// scale factors), M = 128, N = 32, K = 64, A in tensor memory. TMEM lanes 0-63 hold sigma and
// lanes 64-127 tau of the same 64 (stage-matrix, row) pairs: lane 64 p + tm R + r is row r of
// stage-matrix tm = 2 t + matrix (R = 32, 16, 8, 8 rows for T = 1..4), so one MMA covers 64 codes
// of 64 rows and every K position of A carries a code. A code word holds the sigma bits of 16
// codes in its low half and the tau bits in its high half (code i at bit 8 (i % 2) + i / 2); two
// words give one 32-bit register t of sign bits (PRMT of the low or the high halves), and
// register s = ((t << s) & 0x88888888) | 0x22222222 holds eight e2m1 values +-1 (one LOP3).
// x is X = rn(|x| S) < 2^28 (S a power of two per CTA and call) in fourteen base-4 digits d_l,
// each held as the e2m1 value +-d_l / 2 with the sign of x: B row p 14 + l holds digit l of part
// p (re, im) in the K order of A, rows 28-31 are zero. The digit sums are exact in f32 and
// P = (2 / S) sum_l 4^l D_l. Each x entry is off by at most 2^-28 of the largest |x| of the CTA's
// slice of the K range, so the error of x in l1 norm is at most in_features 2^-28 |x|_1
// (<= 9.2e-5 |x|_1 for in_features <= 24576): every output is within 1e-4 |x|_1 sum_t s_t.
//
// Work. A job is one row block (R rows of every stage-matrix) of one linear of a call; a call's
// jobs are dealt round-robin to thread-block clusters of ks CTAs (continuing the deal of the
// previous call), and rank r of a cluster takes the 128-code chunks [r nch / ks, (r+1) nch / ks)
// of every row. A unit is two chunks (one at the end of an odd range) of one job: 4 KB of codes,
// four MMAs. Partial rows are summed in distributed shared memory in rank order (deterministic);
// rank 0 writes y and, once a call's outputs are all written, adds one to the call's completion
// counter in global memory. Before building call c's B tiles a CTA waits (bounded) until call
// c - 1's counter holds every cluster's arrival.
//
// Roles: warps 0-7 are two decoder sets of four (warp w reaches TMEM lanes 32 (w % 4) ..), set s
// decoding units q = s, s + 2, ... into A slot q % 12; warp 8 streams the codes; lane 0 of warps
// 9-16 (issuer e) issues the MMAs of the units v = e, e + 8, ... of every job (counted from a
// rotating start) into the job's accumulator (two buffers, job parity); warps 17-20 and 21-24 are
// two epilogue groups (job parity) that also build the B tiles of every call together.
// A thread blocks for about 150 cycles on each MMA it issues whatever the accumulator, so the
// issue rate grows with the number of issuing warps; all of them add into one accumulator per
// job (the digit sums are exact in f32, so their order does not matter), which the epilogue
// reads and zeroes.
#include <cuda.h>
#include <cuda_bf16.h>

#include <atomic>
#include <mutex>

#include "common.cuh"
#include "ptx.cuh"
#include "tc.cuh"

namespace fairy2i {

namespace ch {

constexpr int kSets = 2;                 // decoder sets of four warps
constexpr int kDecWarps = 4 * kSets;     // warps 0-7
constexpr int kCopyWarp = kDecWarps;     // 8
constexpr int kIss = 8;                  // MMA-issuing threads
constexpr int kIssWarp0 = kCopyWarp + 1; // 9-16
constexpr int kEpiWarp0 = kIssWarp0 + kIss;   // 17-24: two groups of four
constexpr int kBThreads = 256;           // the two epilogue groups build the B tiles
constexpr int kWarps = kEpiWarp0 + 8;
constexpr int kThreads = kWarps * 32;
constexpr int kDigits = 14;
constexpr int kN = 32;                   // MMA N (2 kDigits used)
constexpr int kMaxTok = 4;               // tokens per launch
constexpr int kColAcc = 0;               // accumulators [buffer][token], 32 columns each
constexpr int kColSF = 448;              // unit scale factors
constexpr int kTmemCols = 512;
constexpr int kSlotCols = 32;
constexpr int kUnitBytes = 4096;         // ring slot: one unit's codes
constexpr int kMmaB = kN * 32 + 16;      // B tile of one MMA (+16 B: tiles start in other banks)
constexpr int kChunkB = 2 * kMmaB;
constexpr int kMaxNu = 48;               // chunks of one CTA's K range per call
constexpr int kMaxCluster = 8;
constexpr int kMaxGroup = 4;
constexpr int kMaxCalls = 160;
constexpr int kMaxRing = 48;
constexpr int kSmemLimit = 227 * 1024;
constexpr uint64_t kWaitNs = 1000000000ull;   // 1 s: a pipeline wait is microseconds
constexpr uint32_t kIdesc = idesc_mxf4_f32(128, kN);
constexpr int kBarB = 1, kBarG = 2;      // named barriers: B build (256), epilogue group g (128)
// Tensor-memory plan of a launch with nb tokens: accumulators in columns [0, 64 nb), then the A
// slots (an even number, 32 columns each) up to the scale factors at column 448.
__host__ __device__ constexpr int acc_cols(int nb) { return 64 * nb; }
__host__ __device__ constexpr int num_slots(int nb) { return ((kColSF - acc_cols(nb)) / kSlotCols) & ~1; }
// mbarriers besides the ring's: sfull, sfree per slot; jfull, jfree, gfull, gfree per buffer;
// fin per issuer; sfready
__host__ __device__ constexpr int fixed_bars(int nb) { return 2 * num_slots(nb) + 8 + kIss + 1; }

struct Call {
  const void* x;
  const uint32_t* codes[kMaxGroup];
  const float* scales[kMaxGroup];
  float* y[kMaxGroup];
  int in_features, out_features, n, m;
  int nch;        // 128-code chunks per row
  int rbs;        // row blocks per linear
  int row_tiles;  // ceil(n / 16)
  int G;          // linears sharing x
  int jobs;       // G rbs
  int off;        // cluster that takes job 0
  int xf32;       // x is float32 (else bf16)
  int x_pair;     // pairs of x entries may be loaded as one aligned access
  int x_vec;      // groups of eight bf16 entries may be loaded as one 16-byte access
  int ldx, ldy;   // elements between the tokens of x and of every y
};

struct Args {
  unsigned int* done;     // [ncalls] completion counters, zero on entry (ncalls > 1)
  unsigned int* status;
  int ncalls, ks, ks_shift, nclusters, nring, nu_max;
  Call calls[kMaxCalls];
};

struct Tab {              // per call, this CTA
  int first;              // first job of this cluster
  int nj;                 // jobs of this cluster
  int c0;                 // first chunk of this rank
  int nu;                 // chunks of this rank
};

struct Misc {
  uint32_t tmem;
  int abort;
  unsigned int bprog;     // B tiles built: (build sequence number << 8) | chunks ready
  float xmax[kMaxTok][8];
  float S[kMaxTok], invS[kMaxTok];
  float scl[kMaxGroup][16];
};

struct Smem {             // byte offsets from the 1024-aligned base
  int ring, b, btok, xs, xtok, red, gather, outp, tab, bar, misc, total;
};

// B tiles and bf16 x staging per token (btok, xtok bytes apart), partial outputs per token.
__host__ __device__ inline Smem smem_layout(int nring, int nu_max, int ncalls, int nb) {
  Smem s;
  s.ring = 0;
  s.b = s.ring + nring * kUnitBytes;
  s.btok = (nu_max * kChunkB + 15) & ~15;
  s.xs = s.b + nb * s.btok;
  s.xtok = 2 * 72 * nu_max * 4;         // bf16 x staging: 64 nu words per part + 4 per 32
  s.red = s.xs + nb * s.xtok;
  s.gather = s.red + 2 * 128 * 2 * 4;
  s.outp = s.gather + 2 * kMaxCluster * 64 * nb * 4;
  s.tab = s.outp + 2 * 64 * nb * 4;
  s.bar = s.tab + ncalls * (int)sizeof(Tab);
  s.misc = s.bar + (2 * nring + fixed_bars(nb)) * 8;
  s.total = s.misc + (int)sizeof(Misc) + 1024;   // + alignment slack
  return s;
}

// ---- global-memory completion counters ----
__device__ __forceinline__ unsigned int ld_relaxed_gpu(const unsigned int* p) {
  unsigned int v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void fence_acquire_gpu() {
  asm volatile("fence.acq_rel.gpu;" ::: "memory");
}
__device__ __forceinline__ void red_release_gpu_add(unsigned int* p, unsigned int v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ void bulk_copy_to_cluster(uint32_t dst, uint32_t src, uint32_t bytes,
                                                     uint32_t mbar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(dst), "r"(src), "r"(bytes), "r"(mbar)
      : "memory");
}
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
// Spinning form for the unit pipeline (MMA issuers and decoders): no sleep between tests.
__device__ __forceinline__ bool spin_or_abort(uint64_t* bar, uint32_t parity, volatile int* abort,
                                              unsigned int* status) {
  if (*abort) return false;
  if (mbar_wait_spin(bar, parity, kWaitNs)) return true;
  *abort = 1;
  latch_status(status, kStatusTimeout);
  return false;
}

__device__ __forceinline__ unsigned int ld_acquire_cta(const unsigned int* p) {
  unsigned int v;
  asm volatile("ld.acquire.cta.shared::cta.u32 %0, [%1];" : "=r"(v) : "r"(smem_u32(p)) : "memory");
  return v;
}
__device__ __forceinline__ void st_release_cta(unsigned int* p, unsigned int v) {
  asm volatile("st.release.cta.shared::cta.u32 [%0], %1;" ::"r"(smem_u32(p)), "r"(v) : "memory");
}
// Bounded spin until the B-tile progress word reaches `target` (same build, enough chunks).
__device__ bool wait_bprog(const unsigned int* prog, unsigned int target, volatile int* abort,
                           unsigned int* status) {
  if (ld_acquire_cta(prog) >= target) return true;
  const long long t0 = clock64();
  const long long limit = (long long)(kWaitNs * 5 / 2);
  for (uint32_t i = 0;; ++i) {
    if (ld_acquire_cta(prog) >= target) return true;
    if ((i & 63u) == 63u) {
      if (*abort) return false;
      if (clock64() - t0 > limit) break;
    }
  }
  *abort = 1;
  latch_status(status, kStatusTimeout);
  return false;
}
__device__ __forceinline__ void tmem_ld8(uint32_t taddr, float* v) {
  uint32_t r[8];
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
                 "=r"(r[6]), "=r"(r[7])
               : "r"(taddr)
               : "memory");
#pragma unroll
  for (int i = 0; i < 8; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tmem_ld4(uint32_t taddr, float* v) {
  uint32_t r[4];
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(taddr)
               : "memory");
#pragma unroll
  for (int i = 0; i < 4; ++i) v[i] = __uint_as_float(r[i]);
}

// Bounded wait until *counter >= target (acquire); gives up early once any CTA has latched a
// timeout in the status word.
__device__ bool wait_counter(const unsigned int* counter, unsigned int target, volatile int* abort,
                             unsigned int* status) {
  if (*abort) return false;
  const long long t0 = clock64();
  const long long limit = (long long)(kWaitNs * 5 / 2);
  for (uint32_t i = 0;; ++i) {
    if (ld_relaxed_gpu(counter) >= target) {
      fence_acquire_gpu();   // the counted outputs are visible to this thread's later reads
      return true;
    }
    if ((i & 15u) == 15u) {
      if (*(volatile unsigned int*)status & kStatusTimeout) break;
      if (clock64() - t0 > limit) break;
    }
  }
  *abort = 1;
  latch_status(status, kStatusTimeout);
  return false;
}

// Decoded A registers of one chunk (8 words of a row) for one plane: register 4 q + s holds the
// signs of word pair q (words 2 q, 2 q + 1; low halves for sigma, high halves for tau) at bits
// 4 n + 3 - s, as e2m1 +-1 nibbles.
__device__ __forceinline__ void decode_chunk(const uint32_t (&w)[8], uint32_t sel, uint32_t* r) {
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const uint32_t t = prmt(w[2 * q], w[2 * q + 1], sel);
    r[4 * q + 0] = lop3_and_or(t, 0x88888888u, 0x22222222u);
    r[4 * q + 1] = lop3_and_or(t << 1, 0x88888888u, 0x22222222u);
    r[4 * q + 2] = lop3_and_or(t << 2, 0x88888888u, 0x22222222u);
    r[4 * q + 3] = lop3_and_or(t << 3, 0x88888888u, 0x22222222u);
  }
}

// Two consecutive x entries k, k + 1 of part p of token b (zero past the part's end): float32 x
// as floats, bf16 x as one word (entry k in the low half). Plain loads: x may be an output of
// the previous call, made visible by the completion counter's acquire.
__device__ __forceinline__ float2 load_x_pair_f32(const Call& C, int b, int p, int k) {
  const int lim = p ? C.in_features - C.m : C.m;
  const float* x = static_cast<const float*>(C.x) + (size_t)b * C.ldx + p * C.m;
  float2 v = make_float2(0.f, 0.f);
  if (C.x_pair && k + 1 < lim) {
    v = *reinterpret_cast<const float2*>(x + k);
  } else {
    if (k < lim) v.x = x[k];
    if (k + 1 < lim) v.y = x[k + 1];
  }
  return v;
}
__device__ __forceinline__ float bf_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

template <int T, int NB>
__global__ void __launch_bounds__(kThreads, 1) wl_chain_kernel(const __grid_constant__ Args a) {
  constexpr int kColA = acc_cols(NB);          // A slots, 32 columns each
  constexpr int kSlots = num_slots(NB);        // unit q in slot q % kSlots
  constexpr int kSetSlots = kSlots / kSets;
  static_assert(kSlots >= 2 * kSets && kSlots % kSets == 0, "A slots");
  constexpr int TM = 2 * T;
  constexpr int R = (T == 1) ? 32 : (T == 2 ? 16 : 8);   // rows per row block
  constexpr bool kHalf = R == 8;                          // a job holds half of a 16-row tile
  static_assert(TM * R <= 64, "lanes per plane");
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = align_smem_1024(smem_raw);
  const int ncalls = a.ncalls, nring = a.nring, ks = a.ks;
  const Smem L = smem_layout(nring, a.nu_max, ncalls, NB);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L.bar);
  uint64_t* full = bars;                       // [ring slot] codes landed (tx)
  uint64_t* empty = full + nring;              // [ring slot] codes read (4 warps)
  uint64_t* sfull = empty + nring;             // [slot] A written (4 warps)
  uint64_t* sfree = sfull + kSlots;            // [slot] its MMAs done (1 commit)
  uint64_t* jfull = sfree + kSlots;            // [buffer] job accumulated (every issuer)
  uint64_t* jfree = jfull + 2;                 // [buffer] job read out (4 warps)
  uint64_t* gfull = jfree + 2;                 // [group] rank 0: partials arrived (tx)
  uint64_t* gfree = gfull + 2;                 // [group] ranks > 0: rank 0 read the buffer (1)
  uint64_t* fin = gfree + 2;                   // [issuer] abort path
  uint64_t* sfready = fin + kIss;              // scale factors written (4 warps)
  Misc* misc = reinterpret_cast<Misc*>(smem + L.misc);
  Tab* tab = reinterpret_cast<Tab*>(smem + L.tab);
  volatile int* abort_flag = &misc->abort;
  float* red = reinterpret_cast<float*>(smem + L.red);          // [group][lane][2]
  float* gather = reinterpret_cast<float*>(smem + L.gather);    // [group][rank][token][64]
  float* outp = reinterpret_cast<float*>(smem + L.outp);        // [group][token][64]

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int rank = ks > 1 ? (int)cluster_ctarank() : 0;
  const int cluster = (int)(blockIdx.x >> a.ks_shift);
  const int ncl = a.nclusters;

  // ---- prologue: per-call table, barriers (warp 1), TMEM (warp 0) ----
  for (int c = tid; c < ncalls; c += kThreads) {
    const Call& C = a.calls[c];
    int f = cluster - C.off;
    if (f < 0) f += ncl;
    Tab t;
    t.first = f;
    t.nj = f < C.jobs ? (C.jobs - 1 - f) / ncl + 1 : 0;
    t.c0 = (rank * C.nch) >> a.ks_shift;
    t.nu = (((rank + 1) * C.nch) >> a.ks_shift) - t.c0;
    tab[c] = t;
  }
  if (warp == 1) {
    const int nb = 2 * nring + fixed_bars(NB);
    for (int i = lane; i < nb; i += 32) {
      uint64_t* b = bars + i;
      uint32_t cnt = 1;
      if (b >= empty && b < empty + nring) cnt = 4;
      else if (b >= sfull && b < sfull + kSlots) cnt = 4;
      else if (b == jfull || b == jfull + 1) cnt = kIss;
      else if (b == jfree || b == jfree + 1) cnt = 4;
      else if (b == sfready) cnt = 4;
      mbar_init(b, cnt);
    }
    if (lane == 0) {
      misc->abort = 0;
      misc->bprog = 0;
    }
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&misc->tmem, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = misc->tmem;
  int Q = 0, NJ = 0;   // units and jobs of this CTA over the whole chain
  for (int c = 0; c < ncalls; ++c) {
    Q += tab[c].nj * ((tab[c].nu + 1) >> 1);
    NJ += tab[c].nj;
  }
  if (warp < 4) {
    // Unit scale factors (ue8m0 127 = 1.0) for every row of A and B of every MMA; both
    // accumulators start at zero (every MMA adds).
    uint32_t ones[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) ones[i] = 0x7F7F7F7Fu;
    const uint32_t la = tmem + ((uint32_t)(warp * 32) << 16);
    tmem_st32(la + kColSF, ones);
    tmem_st32(la + kColSF + 32, ones);
#pragma unroll
    for (int i = 0; i < 32; ++i) ones[i] = 0u;
#pragma unroll
    for (int c = 0; c < acc_cols(NB); c += 32) tmem_st32(la + kColAcc + c, ones);
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
    const int Ln = quarter * 32 + lane;
    const int plane = Ln >> 6, j = Ln & 63;
    const uint32_t sel = plane ? 0x7632u : 0x5410u;
    uint32_t lane_off = 0;   // this lane's 32-byte row of chunk 0 inside a ring slot
    if constexpr (kHalf) {
      const int tm = j >> 3, row = j & 7;
      if (tm < TM) lane_off = (uint32_t)(tm * 512 + row * 32);
    } else {
      const int tm = j / R, r = j % R;
      lane_off = (uint32_t)(((tm * (R / 16) + r / 16) * 1024) + (r % 16) * 32);
    }
    const uint32_t chunk1 = kHalf ? 256u : 512u;
    const uint32_t h0 = ((lane >> 2) & 1u) * 16u;   // which 16-byte half first (bank spread)
    const uint32_t ring = smem_u32(smem + L.ring);
    const uint32_t t_lane = tmem + ((uint32_t)(quarter * 32) << 16) + kColA;
    int rs = set, si = set, l = 0;   // ring slot, A slot, units of this set so far
    uint32_t rph = 0, sph = 0;
    if (rs >= nring) { rs -= nring; rph ^= 1u; }
    for (int q = set; q < Q; q += kSets, ++l) {
      if (!__all_sync(0xffffffffu, mbar_test_wait(&full[rs], rph) ||
                                       wait_or_abort(&full[rs], rph, abort_flag, a.status)))
        break;
      const uint32_t src = ring + rs * kUnitBytes + lane_off;
      uint4 v[4];
      v[0] = lds128(src + h0);
      v[1] = lds128(src + (16u - h0));
      v[2] = lds128(src + chunk1 + h0);
      v[3] = lds128(src + chunk1 + (16u - h0));
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[rs]);
      if (l == kSetSlots) pdl_wait_primary();   // later waits depend on MMAs, i.e. on x
      const uint4 a0 = h0 ? v[1] : v[0], a1 = h0 ? v[0] : v[1];
      const uint4 b0 = h0 ? v[3] : v[2], b1 = h0 ? v[2] : v[3];
      const uint32_t w0[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
      const uint32_t w1[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
      uint32_t rr[32];
      decode_chunk(w0, sel, rr);
      decode_chunk(w1, sel, rr + 16);
      // the slot's previous unit has been multiplied (only the store waits for it)
      if (l >= kSetSlots) {
        if (!__all_sync(0xffffffffu, mbar_test_wait(&sfree[si], sph ^ 1u) ||
                                         spin_or_abort(&sfree[si], sph ^ 1u, abort_flag, a.status)))
          break;
        tc_fence_after();
      }
      tmem_st32(t_lane + si * kSlotCols, rr);
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sfull[si]);
      si += kSets;
      if (si >= kSlots) {
        si -= kSlots;
        sph ^= 1u;
      }
      rs += kSets;
      if (rs >= nring) {
        rs -= nring;
        rph ^= 1u;
      }
    }
  } else if (warp == kCopyWarp) {
    // ---------------- code stream: one ring slot per unit ----------------
    const uint64_t pol = l2_evict_first_policy();   // codes are read once per launch
    int q = 0, rs = 0;
    uint32_t use = 0;   // q / nring: unit q is the use-th fill of ring slot rs
    bool ok = true;
    for (int c = 0; ok && c < ncalls; ++c) {
      const Tab tb = tab[c];
      if (tb.nj == 0) continue;
      const Call& C = a.calls[c];
      const int U = (tb.nu + 1) >> 1;
      int g = tb.first / C.rbs, rb = tb.first - g * C.rbs;
      for (int k = 0; ok && k < tb.nj; ++k) {
        for (int v = 0; v < U; ++v, ++q) {
          if (q == nring) pdl_wait_primary();   // refills wait on MMAs, i.e. on x
          if (q >= nring) {
            const bool w =
                lane != 0 || wait_or_abort(&empty[rs], (use - 1u) & 1u, abort_flag, a.status);
            if (!__all_sync(0xffffffffu, w)) {
              ok = false;
              break;
            }
          }
          const int chunks = min(2, tb.nu - 2 * v);
          const int ch0 = tb.c0 + 2 * v;
          const uint32_t* base = C.codes[g];
          unsigned char* dst = smem + L.ring + rs * kUnitBytes;
          if constexpr (kHalf) {
            // every stage-matrix: rows 0-7 or 8-15 of the tile, 256 bytes per chunk
            if (lane == 0) mbar_arrive_expect_tx(&full[rs], (uint32_t)(TM * chunks * 256));
            __syncwarp();
            const int tm = lane >> 1, ch = lane & 1;
            if (tm < TM && ch < chunks) {
              const int64_t tile = (int64_t)tm * C.row_tiles + (rb >> 1);
              bulk_load_hint(dst + tm * 512 + ch * 256,
                             base + (tile * C.nch + ch0 + ch) * 128 + (rb & 1) * 64, 256u,
                             &full[rs], pol);
            }
          } else {
            constexpr int RT = R / 16;   // 16-row tiles per stage-matrix and job
            int nrt = 0;                 // tiles of the row block that exist
#pragma unroll
            for (int k2 = 0; k2 < RT; ++k2) nrt += (rb * RT + k2 < C.row_tiles) ? 1 : 0;
            if (lane == 0) mbar_arrive_expect_tx(&full[rs], (uint32_t)(TM * nrt * chunks * 512));
            __syncwarp();
            const int tm = lane / RT, rt = lane % RT;
            if (lane < TM * RT && rt < nrt) {
              const int64_t tile = (int64_t)tm * C.row_tiles + rb * RT + rt;
              bulk_load_hint(dst + lane * 1024, base + (tile * C.nch + ch0) * 128,
                             (uint32_t)(chunks * 512), &full[rs], pol);
            }
          }
          if (++rs == nring) {
            rs = 0;
            ++use;
          }
        }
        rb += ncl;
        while (rb >= C.rbs) {
          rb -= C.rbs;
          ++g;
        }
      }
    }
    // Abort path: every issued copy lands before shared memory is released.
    if (lane == 0 && *abort_flag) {
      for (int i = (q > nring ? q - nring : 0); i < q; ++i)
        (void)mbar_wait_timed(&full[i % nring], (i / nring) & 1, 1000000ull);
    }
  } else if (warp < kEpiWarp0) {
    // ---- MMA issuers: lane 0 of warp kIssWarp0 + e (e < kIssN) issues unit v of a job when
    // (v + r) % kIssN == e, r = the units of this CTA before the job; unit q (counted over the
    // whole chain) sits in A slot q % kSlots. An issuer reaches unit q only after unit
    // q - kIssN was written, hence (kIssN <= kSlots, same decoder set, decoded in order) after
    // unit q - kSlots: the slot's barrier is never two phases behind its waiter. ----
    constexpr int kIssN = kIss < kSlots ? kIss : kSlots;
    const int e = warp - kIssWarp0;
    if (lane == 0) {
      const uint32_t b_base = smem_u32(smem + L.b);
      const uint64_t desc0 = smem_desc(b_base, 128, 256);
      pdl_wait_primary();
      bool ok = wait_or_abort(sfready, 0, abort_flag, a.status);
      bool issued = false;
      int J = 0, qb = 0;   // jobs and units before the current job
      uint32_t seq = 0;
      for (int c = 0; ok && c < ncalls; ++c) {
        const Tab tb = tab[c];
        if (tb.nj == 0) continue;
        const int U = (tb.nu + 1) >> 1;
        ++seq;   // this call's B tiles are the seq-th build; unit v needs its chunks built
        int have = 0;
        for (int k = 0; ok && k < tb.nj; ++k, ++J, qb += U) {
          const int buf = J & 1;
          // the read-out of job J - 2 (same buffer) is done and its accumulators zeroed
          if (J >= 2) ok = wait_or_abort(&jfree[buf], ((J >> 1) - 1) & 1, abort_flag, a.status);
          if (!ok) break;
          tc_fence_after();
          int v0 = (e - qb) % kIssN;
          if (v0 < 0) v0 += kIssN;
          if (e < kIssN && v0 < U) {
            const uint32_t d0 = tmem + kColAcc + (uint32_t)(buf * NB * 32);
            for (int v = v0, q = qb + v0; v < U; v += kIssN, q += kIssN) {
              const int si = q % kSlots;
              const uint32_t sph = (uint32_t)(q / kSlots) & 1u;
              const int need = min(tb.nu, 2 * v + 2);
              if (have < need) {
                ok = wait_bprog(&misc->bprog, (seq << 8) | (uint32_t)need, abort_flag, a.status);
                if (!ok) break;
                have = need;
              }
              ok = mbar_test_wait(&sfull[si], sph) ||
                   spin_or_abort(&sfull[si], sph, abort_flag, a.status);
              if (!ok) break;
              tc_fence_after();
              const uint32_t a_slot = tmem + kColA + (uint32_t)(si * kSlotCols);
              const int nm = 2 * min(2, tb.nu - 2 * v);
#pragma unroll
              for (int b = 0; b < NB; ++b) {
                // token b's B tiles, btok bytes after token b - 1's (a multiple of 16)
                const uint64_t bd = desc0 + (uint64_t)((b * L.btok + 4 * v * kMmaB) >> 4);
#pragma unroll
                for (int jm = 0; jm < 4; ++jm)
                  if (jm < nm)
                    mma_mxf4_ts(d0 + b * 32, a_slot + jm * 8, bd + (uint64_t)((jm * kMmaB) >> 4),
                                kIdesc, tmem + kColSF, tmem + kColSF + 16, 1u);
              }
              issued = true;
              mma_commit(&sfree[si]);
            }
            if (!ok) break;
            mma_commit(&jfull[buf]);
          } else {
            mbar_arrive(&jfull[buf]);
          }
        }
      }
      // Abort path: the MMAs this thread issued finish before TMEM is released.
      if (issued && *abort_flag) {
        mma_commit(&fin[e]);
        (void)mbar_wait_timed(&fin[e], 0, kWaitNs);
      }
    }
    __syncwarp();
  } else {
    // ------ epilogue groups: B tiles of every call, then the read-out of every job ------
    const int bt = tid - kEpiWarp0 * 32;          // 0 .. 255
    const int grp = (warp - kEpiWarp0) >> 2;       // job parity
    const int et = bt - grp * 128;                 // 0 .. 127 inside the group
    const int quarter = warp & 3;
    const int Ln = quarter * 32 + lane;
    // Rows 28-31 of every B tile of every token stay zero.
    for (int o = bt; o < NB * a.nu_max * 2 * 4 * 2; o += kBThreads) {
      const int tb_ = o / (a.nu_max * 16), oo = o - tb_ * (a.nu_max * 16);
      const int tile = oo >> 3, rest = oo & 7, nrow = 2 * kDigits + (rest >> 1);
      *reinterpret_cast<uint4*>(smem + L.b + tb_ * L.btok + tile * kMmaB + (nrow >> 3) * 256 +
                                (rest & 1) * 128 + (nrow & 7) * 16) = make_uint4(0, 0, 0, 0);
    }
    pdl_wait_primary();   // x may be written, and y read, by the previous kernel
    if (ks > 1) cluster_wait();   // every rank's barriers are initialised
    int nbuilt = 0, J = 0;
    for (int c = 0; c < ncalls; ++c) {
      const Tab tb = tab[c];
      const Call& C = a.calls[c];
      if (tb.nj > 0) {
        // -------- B tiles of call c: after every output of call c - 1 is written --------
        // While the previous call finishes, warm L2 with this CTA's slice of x: a prefetch
        // returns nothing to the program, so it may precede the dependency wait (L2 is the
        // point of coherence of global memory).
        if (bt < 2 * NB) {
          const int pp = bt & 1, tk = bt >> 1;
          const int lim = pp ? C.in_features - C.m : C.m;
          const int k0 = 128 * tb.c0, k1 = min(128 * (tb.c0 + tb.nu), lim);
          if (k1 > k0) {
            const int esz = C.xf32 ? 4 : 2;
            const uintptr_t b0 = reinterpret_cast<uintptr_t>(C.x) +
                                 ((size_t)tk * C.ldx + (size_t)pp * C.m + k0) * esz;
            const uintptr_t a0 = (b0 + 15) & ~uintptr_t(15);
            const uintptr_t a1 = (b0 + (size_t)(k1 - k0) * esz) & ~uintptr_t(15);
            if (a1 > a0) prefetch_l2_bulk(reinterpret_cast<const void*>(a0), (uint32_t)(a1 - a0));
          }
        }
        if (bt == 0) {
          if (c > 0 && a.done) (void)wait_counter(a.done + (c - 1), (unsigned)ncl, abort_flag, a.status);
        }
        named_bar_sync(kBarB, kBThreads);
        // Pass 1: max |x| over the slice, per token; bf16 x is staged in shared memory by
        // 16-byte loads (word w of a part at w + 4 (w / 32): the pass-2 reads of a warp hit 32
        // banks), float32 x is read twice from global memory.
        const bool f32 = C.xf32 != 0;
        const int nv = 16 * tb.nu;        // groups of eight entries per part
        const int pw = 72 * a.nu_max;      // staging words per part
        float mx[NB];
#pragma unroll
        for (int b = 0; b < NB; ++b) mx[b] = 0.f;
#pragma unroll
        for (int b = 0; b < NB; ++b) {
          uint32_t* xs = reinterpret_cast<uint32_t*>(smem + L.xs + b * L.xtok);
          for (int i = bt; i < 2 * nv; i += kBThreads) {
            const int p = i >= nv ? 1 : 0, v = i - p * nv;
            const int lim = p ? C.in_features - C.m : C.m;
            const int k = 128 * tb.c0 + 8 * v;
            if (!f32) {
              const unsigned short* xp =
                  static_cast<const unsigned short*>(C.x) + (size_t)b * C.ldx + p * C.m;
              uint4 q;
              if (C.x_vec && k + 8 <= lim) {
                q = *reinterpret_cast<const uint4*>(xp + k);
              } else {
                uint32_t h[8];
#pragma unroll
                for (int z = 0; z < 8; ++z) h[z] = k + z < lim ? (uint32_t)xp[k + z] : 0u;
                q = make_uint4(h[0] | (h[1] << 16), h[2] | (h[3] << 16), h[4] | (h[5] << 16),
                               h[6] | (h[7] << 16));
              }
              const uint32_t ww[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
              for (int z = 0; z < 4; ++z)
                mx[b] = fmaxf(mx[b], fmaxf(fabsf(bf_lo(ww[z])), fabsf(bf_hi(ww[z]))));
              *reinterpret_cast<uint4*>(xs + p * pw + 4 * v + 4 * (v >> 3)) = q;
            } else {
#pragma unroll
              for (int z = 0; z < 8; z += 2) {
                const float2 f = load_x_pair_f32(C, b, p, k + z);
                mx[b] = fmaxf(mx[b], fmaxf(fabsf(f.x), fabsf(f.y)));
              }
            }
          }
        }
#pragma unroll
        for (int b = 0; b < NB; ++b) {
#pragma unroll
          for (int o = 16; o >= 1; o >>= 1) mx[b] = fmaxf(mx[b], __shfl_xor_sync(0xffffffffu, mx[b], o));
          if (lane == 0) misc->xmax[b][bt >> 5] = mx[b];
        }
        if (bt < C.G * 4 * T) {
          const int gl = bt / (4 * T), idx = bt - gl * 4 * T;
          misc->scl[gl][idx] = C.scales[gl][idx];
        }
        named_bar_sync(kBarB, kBThreads);
        // S = 2^(28 - E) for 2^(E-1) <= max|x| < 2^E (per token): every X = rn(|x| S) < 2^28
        float Sb[NB];
#pragma unroll
        for (int b = 0; b < NB; ++b) {
          float xm = misc->xmax[b][0];
#pragma unroll
          for (int w = 1; w < 8; ++w) xm = fmaxf(xm, misc->xmax[b][w]);
          const int ef = (int)((__float_as_uint(xm) >> 23) & 0xffu);
          const int se = max(1, min(254, 281 - ef));
          Sb[b] = __uint_as_float((uint32_t)se << 23);
        }
        // Pass 2. Task t: lane ln = s' + 4 (tile % 8) of group (tile / 8, pair, part): B column
        // 4 pair + s' of tile (chunk u, MMA hw), rows p 14 + l. Its eight values (nibble n) are
        // codes 2(3-s'), 2(7-s'), 2(3-s')+1, 2(7-s')+1 of words 4 hw + 2 pair and + 1, i.e. the
        // entry pairs at k, k + 8, k + 16, k + 24 (k = 128 u + 64 hw + 32 pair + 2 (3 - s')).
        // X = rn(|x| S) of the eight values, transposed as an 8 x 8 nibble matrix, gives in word
        // j the nibble j (digits 2 j, 2 j + 1) of every value.
        // Every round of 256 tasks completes eight chunks, which are published at once (MMAs of
        // the first units start while the later chunks are built).
        if (bt < NB) {
          misc->S[bt] = Sb[bt];
          misc->invS[bt] = 2.f / Sb[bt];
        }
        const uint32_t seq = (uint32_t)(nbuilt + 1) << 8;
        const int ntask = 128 * ((2 * tb.nu + 7) >> 3);
        for (int t0 = 0; t0 < ntask; t0 += kBThreads) {
          const int t = t0 + bt;
          const int ln = t & 31, sp = ln & 3, tile = ((t >> 7) << 3) + (ln >> 2);
          const int pair = (t >> 6) & 1, p = (t >> 5) & 1;
#pragma unroll 1
          for (int b = 0; b < NB; ++b) {
          if (t >= ntask || tile >= 2 * tb.nu) break;
          const int u = tile >> 1, hw = tile & 1;
          const float S = Sb[b];
          float2 pv[4];
          if (!f32) {
            const uint32_t* xs = reinterpret_cast<const uint32_t*>(smem + L.xs + b * L.xtok);
            const int w0 = 64 * u + 32 * hw + 16 * pair + 3 - sp;
#pragma unroll
            for (int h = 0; h < 4; ++h) {
              const int w = w0 + 4 * h;
              const uint32_t q = xs[p * pw + w + 4 * (w >> 5)];
              pv[h] = make_float2(bf_lo(q), bf_hi(q));
            }
          } else {
            const int k = 128 * (tb.c0 + u) + 64 * hw + 32 * pair + 2 * (3 - sp);
#pragma unroll
            for (int h = 0; h < 4; ++h) pv[h] = load_x_pair_f32(C, b, p, k + 8 * h);
          }
          // nibble n: n = 0: pair 0 lo, 1: pair 1 lo, 2: pair 0 hi, 3: pair 1 hi, 4-7: +16
          const float vals[8] = {pv[0].x, pv[1].x, pv[0].y, pv[1].y,
                                 pv[2].x, pv[3].x, pv[2].y, pv[3].y};
          uint32_t X[8], sg = 0u;
#pragma unroll
          for (int n = 0; n < 8; ++n) {
            X[n] = __float2uint_rn(fabsf(vals[n]) * S);
            sg |= (__float_as_uint(vals[n]) >> 31) << (4 * n + 3);
          }
          transpose_nibbles(X);
          unsigned char* col = smem + L.b + b * L.btok + tile * kMmaB + pair * 128 + sp * 4;
#pragma unroll
          for (int l = 0; l < kDigits; ++l) {
            const uint32_t w = lop3_and_or(X[l >> 1] >> (2 * (l & 1)), 0x33333333u, sg);
            const int nrow = p * kDigits + l;
            *reinterpret_cast<uint32_t*>(col + (nrow >> 3) * 256 + (nrow & 7) * 16) = w;
          }
          }
          fence_proxy_async_smem();   // generic-proxy writes of B visible to the tensor cores
          named_bar_sync(kBarB, kBThreads);
          if (bt == 0) st_release_cta(&misc->bprog, seq | (uint32_t)min(tb.nu, (t0 >> 5) + 8));
        }
        ++nbuilt;
        float invS[NB];
#pragma unroll
        for (int b = 0; b < NB; ++b) invS[b] = misc->invS[b];

        // -------- the jobs of call c: group grp reads out the jobs of its parity --------
        int g = tb.first / C.rbs, rb = tb.first - g * C.rbs;
        for (int k = 0; k < tb.nj; ++k, ++J) {
          if ((J & 1) == grp) {
            const int jg = J >> 1;
            const bool got = __all_sync(0xffffffffu,
                                        wait_or_abort(&jfull[grp], jg & 1, abort_flag, a.status));
            tc_fence_after();
            float vre[NB], vim[NB];
#pragma unroll
            for (int b = 0; b < NB; ++b) vre[b] = vim[b] = 0.f;
            if (got) {
              // per token: the 28 digit columns (loads of 16 + 8 + 4, one wait), then zeroes
              // for the job after next
#pragma unroll
              for (int b = 0; b < NB; ++b) {
                const uint32_t ta = tmem + ((uint32_t)(quarter * 32) << 16) + kColAcc +
                                    (uint32_t)((grp * NB + b) * 32);
                float d[28];
                tmem_ld16(ta, *reinterpret_cast<float(*)[16]>(&d[0]));
                tmem_ld8(ta + 16, &d[16]);
                tmem_ld4(ta + 24, &d[24]);
                tmem_wait_ld();
#pragma unroll
                for (int l = 0; l < kDigits; ++l) {
                  const float wgt = (float)(1u << (2 * l));
                  vre[b] = fmaf(d[l], wgt, vre[b]);
                  vim[b] = fmaf(d[kDigits + l], wgt, vim[b]);
                }
                tmem_zero16(ta);
                tmem_zero16(ta + 16);
              }
              tmem_wait_st();
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&jfree[grp]);
            // row r, component comp of token b: sum over the stage-matrices of h P + conj(h) Q
            // (U) or h conj(P) + conj(h) conj(Q) (W)
            float* rg = red + grp * 256;
            float val[NB];
#pragma unroll
            for (int b = 0; b < NB; ++b) {
              rg[Ln * 2 + 0] = vre[b] * invS[b];
              rg[Ln * 2 + 1] = vim[b] * invS[b];
              named_bar_sync(kBarG + grp, 128);
              val[b] = 0.f;
              if (et < 2 * R) {
                const int r = et >> 1, comp = et & 1;
#pragma unroll
                for (int tm = 0; tm < TM; ++tm) {
                  const float pre = rg[(tm * R + r) * 2], qre = rg[(64 + tm * R + r) * 2];
                  float pim = rg[(tm * R + r) * 2 + 1], qim = rg[(64 + tm * R + r) * 2 + 1];
                  if (tm & 1) {
                    pim = -pim;
                    qim = -qim;
                  }
                  const float hr = 0.5f * misc->scl[g][tm * 2 + 0];
                  const float hi = 0.5f * misc->scl[g][tm * 2 + 1];
                  val[b] += comp == 0 ? hr * (pre + qre) - hi * (pim - qim)
                                      : hr * (pim + qim) + hi * (pre - qre);
                }
              }
              named_bar_sync(kBarG + grp, 128);   // red is free for the next token or job
            }
            bool write = rank == 0;
            if (ks > 1) {
              // partial rows of every token (64 floats each) go to rank 0 in one bulk copy
              if (rank != 0) {
                const bool fr = jg < 1 ||
                                __all_sync(0xffffffffu, wait_or_abort(&gfree[grp], (jg - 1) & 1,
                                                                      abort_flag, a.status));
                const bool ok2 = fr && !*abort_flag;
                float* op = outp + grp * 64 * NB;
#pragma unroll
                for (int b = 0; b < NB; ++b)
                  if (et < 2 * R) op[b * 64 + et] = ok2 ? val[b] : 0.f;
                fence_proxy_async_smem();
                named_bar_sync(kBarG + grp, 128);
                if (et == 0) {
                  const uint32_t g0 =
                      smem_u32(gather) + (uint32_t)((grp * kMaxCluster + rank) * 64 * NB) * 4;
                  bulk_copy_to_cluster(mapa_shared(g0, 0), smem_u32(op), (uint32_t)(64 * NB * 4),
                                       mapa_shared(smem_u32(&gfull[grp]), 0));
                  bulk_commit_wait_read();
                }
              } else {
                if (et == 0)
                  mbar_arrive_expect_tx(&gfull[grp], (uint32_t)((ks - 1) * 64 * NB * 4));
                const bool got2 =
                    __all_sync(0xffffffffu, mbar_wait_cluster_poll(&gfull[grp], jg & 1, kWaitNs)) &&
                    !*abort_flag;
                if (!got2) {
                  if (!*abort_flag) {
                    *abort_flag = 1;
                    latch_status(a.status, kStatusTimeout);
                  }
                  write = false;
                } else if (et < 2 * R) {
                  for (int r2 = 1; r2 < ks; ++r2)
#pragma unroll
                    for (int b = 0; b < NB; ++b)
                      val[b] += gather[((grp * kMaxCluster + r2) * NB + b) * 64 + et];
                }
                named_bar_sync(kBarG + grp, 128);   // every read of gather[grp] is done
                // Rank r waits for this release only before this group's next job, so the last
                // job of the group sends none: no remote access reaches an exited CTA.
                if (et < ks - 1 && J + 2 < NJ)
                  mbar_arrive_remote(mapa_shared(smem_u32(&gfree[grp]), et + 1));
              }
            }
            if (write && !*abort_flag && et < 2 * R) {
              const int r = et >> 1, comp = et & 1;
              const int jr = rb * R + r;
              if (jr < C.n) {
#pragma unroll
                for (int b = 0; b < NB; ++b) {
                  float* yg = C.y[g] + (size_t)b * C.ldy;
                  if (comp == 0) yg[jr] = val[b];
                  else if (C.n + jr < C.out_features) yg[C.n + jr] = val[b];
                }
              }
            }
          }
          rb += ncl;
          while (rb >= C.rbs) {
            rb -= C.rbs;
            ++g;
          }
        }
      }
      // -------- call c complete on this CTA: rank 0 counts it once its outputs are visible ----
      if (a.done) {
        // Every y store of this CTA precedes the barrier; one thread's device-scope release
        // then orders them (cumulatively) before the counter update.
        named_bar_sync(kBarB, kBThreads);
        if (bt == 0 && rank == 0 && !*abort_flag) red_release_gpu_add(a.done + c, 1u);
      }
    }
  }

  // Teardown. The first cluster barrier was waited by the epilogue warps; every other thread
  // waits it here.
  if (ks > 1 && warp < kEpiWarp0) cluster_wait();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0) tmem_dealloc(tmem, kTmemCols);
}

template <int T, int NB>
fairy2i_status launch(const Args& a, int grid, int smem, cudaStream_t stream) {
  auto kern = wl_chain_kernel<T, NB>;
  static std::atomic<uint64_t> smem_set{0};
  if (!smem_attr_once(kern, kSmemLimit, smem_set)) return FAIRY2I_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = (size_t)smem;
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

// Clusters of `ks` CTAs (one per SM) that can be resident at once on the device (0 if none).
template <int T, int NB>
int max_clusters(int ks) {
  auto kern = wl_chain_kernel<T, NB>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit) !=
      cudaSuccess)
    return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(ks * 256));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmemLimit;
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

// Tokens per launch the kernel is built for: 1 to 4.
inline int tok_index(int nb) { return nb - 1; }

template <int NB>
int max_clusters_t(int T, int ks) {
  switch (T) {
    case 1: return max_clusters<1, NB>(ks);
    case 2: return max_clusters<2, NB>(ks);
    case 3: return max_clusters<3, NB>(ks);
    case 4: return max_clusters<4, NB>(ks);
  }
  return 0;
}

template <int NB>
fairy2i_status launch_t(int T, const Args& a, int grid, int smem, cudaStream_t stream) {
  switch (T) {
    case 1: return launch<1, NB>(a, grid, smem, stream);
    case 2: return launch<2, NB>(a, grid, smem, stream);
    case 3: return launch<3, NB>(a, grid, smem, stream);
    case 4: return launch<4, NB>(a, grid, smem, stream);
  }
  return FAIRY2I_ERR_INVALID_ARG;
}

}  // namespace ch

namespace {
std::mutex g_ch_mu;
int g_ch_clusters[64][4][4][4];   // [device][ks index][T - 1][tokens - 1], -1 = unknown
bool g_ch_init[64];
}  // namespace

static int ch_resident_clusters(int dev, int ks_idx, int T, int nb) {
  std::lock_guard<std::mutex> lock(g_ch_mu);
  if (!g_ch_init[dev]) {
    for (int i = 0; i < 4; ++i)
      for (int t = 0; t < 4; ++t)
        for (int b = 0; b < 4; ++b) g_ch_clusters[dev][i][t][b] = -1;
    g_ch_init[dev] = true;
  }
  int& v = g_ch_clusters[dev][ks_idx][T - 1][ch::tok_index(nb)];
  if (v < 0) {
    const int ks = 1 << ks_idx;
    switch (nb) {
      case 1: v = ch::max_clusters_t<1>(T, ks); break;
      case 2: v = ch::max_clusters_t<2>(T, ks); break;
      case 3: v = ch::max_clusters_t<3>(T, ks); break;
      case 4: v = ch::max_clusters_t<4>(T, ks); break;
      default: v = 0;
    }
  }
  return v;
}

int chain_max_calls() { return ch::kMaxCalls; }

// Checks the calls against the kernel's limits (nb = 1 to 4 tokens per call, x float32 or
// bf16, T <= 4, in_features <= 24576) and launches. Token b of call c reads x + b ldx and writes
// y[g] + b ldy (elements; ignored for nb = 1). `done` holds ncalls zeroed counters (unused for
// one call); cluster_size 0 picks the cluster size, else 1, 2, 4 or 8.
fairy2i_status launch_wl_chain(const fairy2i_chain_call* calls, int ncalls, int T,
                               int cluster_size, unsigned int* done, cudaStream_t stream, int nb,
                               int64_t ldx, int64_t ldy) {
  using namespace ch;
  if (ncalls < 1 || ncalls > kMaxCalls || T < 1 || T > 4) return FAIRY2I_ERR_INVALID_ARG;
  if (nb < 1 || nb > kMaxTok) return FAIRY2I_ERR_INVALID_ARG;
  if (nb == 1) ldx = ldy = 0;
  if (ldx < 0 || ldy < 0 || ldx > (int64_t(1) << 30) || ldy > (int64_t(1) << 30))
    return FAIRY2I_ERR_INVALID_ARG;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return FAIRY2I_ERR_CUDA;
  int sms = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
    return FAIRY2I_ERR_CUDA;
  const int R = T == 1 ? 32 : (T == 2 ? 16 : 8);
  int nch_min = 1 << 30, nch_max = 0;
  for (int c = 0; c < ncalls; ++c) {
    const int64_t m = (calls[c].in_features + 1) / 2;
    const int nch = (int)((m + 127) / 128);
    nch_min = std::min(nch_min, nch);
    nch_max = std::max(nch_max, nch);
  }
  if (nch_max > 8 * kMaxNu || nch_max > 192) return FAIRY2I_ERR_INVALID_ARG;
  // Cluster size: every rank needs a chunk and at most kMaxNu of them, and the B tiles of nb
  // tokens (with a ring of at least four units) must fit in shared memory; among the sizes that
  // fit, the automatic choice minimises an estimate of the busiest cluster's time per call:
  // jobs x (units + an epilogue of about half a unit) + a quarter unit of B tiles per chunk,
  // the MMA and B-tile terms growing with the tokens.
  int best_ks = 0, best_ncl = 0;
  double best_cost = 0.0;
  for (int ki = 0; ki < 4; ++ki) {
    const int ks = 1 << ki;
    if (cluster_size != 0 && ks != cluster_size) continue;
    const int nu_max = (nch_max + ks - 1) / ks;
    if (nch_min < ks || nu_max > kMaxNu) continue;
    if (smem_layout(4, nu_max, ncalls, nb).total > kSmemLimit) continue;
    const int ncl = std::min(ch_resident_clusters(dev, ki, T, nb), sms / ks);
    if (ncl < 1) continue;
    double cost = 0.0;
    for (int c = 0; c < ncalls; ++c) {
      const int64_t n = (calls[c].out_features + 1) / 2, m = (calls[c].in_features + 1) / 2;
      const int64_t nch = (m + 127) / 128, nu = (nch + ks - 1) / ks;
      const int64_t jobs = calls[c].count * ((n + R - 1) / R);
      const int64_t per = (jobs + ncl - 1) / ncl;
      cost += (double)per * (double)(nb * (nu + 1) / 2 + 0.5) + 0.25 * nb * (double)nu + 4.0;
    }
    if (best_ks == 0 || cost < best_cost) {
      best_cost = cost;
      best_ks = ks;
      best_ncl = ncl;
    }
  }
  if (best_ks == 0) return FAIRY2I_ERR_INVALID_ARG;
  Args a;
  a.done = ncalls > 1 ? done : nullptr;
  a.status = device_status_word();
  a.ncalls = ncalls;
  a.ks = best_ks;
  a.ks_shift = best_ks == 1 ? 0 : (best_ks == 2 ? 1 : (best_ks == 4 ? 2 : 3));
  a.nclusters = best_ncl;
  a.nu_max = (nch_max + best_ks - 1) / best_ks;
  int64_t deal = 0;
  for (int c = 0; c < ncalls; ++c) {
    const fairy2i_chain_call& in = calls[c];
    Call& C = a.calls[c];
    const int64_t n = (in.out_features + 1) / 2, m = (in.in_features + 1) / 2;
    C.x = in.x;
    for (int g = 0; g < kMaxGroup; ++g) {
      const int gg = g < in.count ? g : 0;
      C.codes[g] = in.codes[gg];
      C.scales[g] = in.scales[gg];
      C.y[g] = in.y[gg];
    }
    C.in_features = (int)in.in_features;
    C.out_features = (int)in.out_features;
    C.n = (int)n;
    C.m = (int)m;
    C.nch = (int)((m + 127) / 128);
    C.rbs = (int)((n + R - 1) / R);
    C.row_tiles = (int)((n + 15) / 16);
    C.G = in.count;
    C.jobs = in.count * C.rbs;
    C.off = (int)(deal % best_ncl);
    deal += C.jobs;
    C.xf32 = in.xdt == FAIRY2I_F32 ? 1 : 0;
    C.ldx = (int)ldx;
    C.ldy = (int)ldy;
    // wide loads where every token's parts keep their alignment
    const uintptr_t xa = reinterpret_cast<uintptr_t>(in.x);
    C.x_pair = (m % 2 == 0 && ldx % 2 == 0 && xa % 8 == 0) ? 1 : 0;
    C.x_vec = (m % 8 == 0 && ldx % 8 == 0 && xa % 16 == 0) ? 1 : 0;
  }
  // The code ring takes the shared memory the rest leaves.
  const Smem base = smem_layout(0, a.nu_max, ncalls, nb);
  a.nring = std::min(kMaxRing, (kSmemLimit - base.total - 2 * 8) / (kUnitBytes + 16));
  if (a.nring < 4) return FAIRY2I_ERR_INVALID_ARG;
  const Smem lay = smem_layout(a.nring, a.nu_max, ncalls, nb);
  if (lay.total > kSmemLimit) return FAIRY2I_ERR_INVALID_ARG;
  const int grid = best_ncl * best_ks;
  switch (nb) {
    case 1: return launch_t<1>(T, a, grid, lay.total, stream);
    case 2: return launch_t<2>(T, a, grid, lay.total, stream);
    case 3: return launch_t<3>(T, a, grid, lay.total, stream);
    case 4: return launch_t<4>(T, a, grid, lay.total, stream);
  }
  return FAIRY2I_ERR_INVALID_ARG;
}

}  // namespace fairy2i
