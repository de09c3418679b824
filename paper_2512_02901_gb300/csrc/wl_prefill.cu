// Prefill (many-token) kernel of the quantized widely-linear matmul on the 5th-generation tensor
// cores: a GEMM whose weight operand is expanded from the 2-bit codes on the fly.
//
// Arithmetic (Eq. ifairy-dequant, Algorithm 1 with the W conj(x) term): with sigma = sign(Re b +
// Im b), tau = sign(Re b - Im b) of the codeword b and h = (s_re + i s_im)/2, the dequantized
// weight is h sigma + conj(h) tau, so per (stage t, matrix) and output row the layer needs the +-1
// sums P = sum_k sigma_k x_k and Q = sum_k tau_k x_k; y += h P + conj(h) Q for U and
// h conj(P) + conj(h) conj(Q) for W. +-1 and bf16 x are exact in a bf16 x bf16 -> f32 MMA.
//
// GEMM form. Tile = one row block (R rows of every stage-matrix: TMEM lane tm*R + r, R = 64, 32,
// 16, 16 for T = 1..4) x 64 tokens. Per 16 codes (one code word per lane) two tcgen05.mma
// kind::f16 (M = 128, N = 128, K = 16) run: A = the sigma (or tau) plane of the word as bf16 +-1 in
// tensor memory, B = x of the 64 tokens (rows 0-63: Re x, rows 64-127: Im x) in shared memory, D =
// the sigma accumulator (TMEM columns 0-127) or the tau accumulator (128-255): column p*64 + b is
// the sum for part p (re/im) of token b. x arrives by TMA (128-byte swizzle, boxes of 64 codes x
// 64 tokens per part; Re and Im through two tensor maps so that each part is zero beyond its end).
// The CTAs are persistent over the tiles, ordered token-tile-major so that CTAs running together
// share x in L2.
//
// Pipeline granularity: a group = 64 codes = 4 steps of 16 codes = 2 step pairs. The A ring holds
// 4 groups (64 TMEM columns each); an x stage holds 128 codes (two groups), which the decoders
// take per iteration. Per group an issuer makes one barrier wait (the group's full barrier, which
// the decoders complete once the A pairs are stored and x has landed) and one commit (plus one
// per x stage): the issue cost per MMA is what bounds this kernel once the waits are per MMA.
//
// Roles (16 warps, 18 at 32-token tiles; warp w reaches TMEM lanes 32 (w % 4) ..): warps 0-7,
// two sets of four, decode the code words into the A ring, set s taking pair s of every group
// (one 32-column store: sigma, tau of two steps, left in flight while the next group is decoded),
// warp 0 also relaying the x-stage arrival into the group barrier; they run on into the next
// tile without a pause. Warps
// 8 and 9 issue the sigma and the tau MMAs (8-11 at 32-token tiles); the next warp copies x in
// (TMA) and the one after it the codes (bulk copies of whole 16-row tiles), each on its own since
// a thread blocks for a while on every copy it issues; the last four run the epilogue of each tile
// (every accumulator column is read out first, so the MMAs of the next tile start before the
// reduction and the stores).
//
// K split over CTA pairs. When the tiles fill the SMs poorly (a few tiles per SM, as at batches of
// up to 64 tokens: 64 tiles of an attention output projection on 152 SMs) the launch is made of
// clusters of two CTAs that work the same tile on the two halves of its 128-code chunks. Rank 1
// sums its partials over the stage-matrices, packs the sums in its reduction buffer and arrives
// (release, cluster scope) on rank 0's barrier; rank 0 reads them over distributed shared memory
// and stores its own sum + rank 1's, always in that order, so the result does not depend on
// timing. Rank 0 returns a credit per tile before rank 1 overwrites the buffer with the next one.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>

#include <mutex>

#include "common.cuh"
#include "ptx.cuh"
#include "tc.cuh"

namespace fairy2i {

namespace pfl {

constexpr int kIssWarp = 8;                       // warps 0-7 decode, then the MMA issuers
constexpr int kG = 4;                             // A ring: groups of 64 codes (4 steps)
constexpr int kColD = 0;                          // accumulators [plane][issuer], 256 columns
constexpr int kColA = 256;                        // A ring: 64 columns per group
constexpr int kTmemCols = 512;
constexpr int kXS = 4;                            // x stages
constexpr int kCChunks = 2;                       // 128-code chunks per code stage (4 groups)
constexpr int kCS = 3;                            // code stages
constexpr int kCStage = kCChunks * 8 * 512;       // <= 8 tiles x kCChunks x 512 B
constexpr int kGroupsPerCStage = 2 * kCChunks;
constexpr int kRed = 4 * 16 * 2 * 128;            // floats: [sub-block][16 tokens][2][128 lanes]
constexpr uint64_t kWaitNs = 1000000000ull;

// Token-tile forms. TOK = 64: N = 128, one issuing thread per sign plane (each blocks ~200 cycles
// on an MMA that keeps the tensor pipe ~64 cycles busy: the issue rate bounds the MMA phase; the
// accumulators of more issuing threads would not leave tensor memory for the A ring).
// TOK = 32 (batches of at most 32 tokens): N = 64, two issuing threads per plane taking
// alternate groups, each into its own accumulator (an issuing thread blocks for about 150 cycles
// on every MMA, so at the smaller N the issue rate is the bound); the epilogue adds the two in a
// fixed order, so the result is deterministic.
template <int TOK>
struct Cfg {
  static constexpr int kIssPP = TOK == 32 ? 2 : 1;          // issuing threads per sign plane
  static constexpr int kIssN = 2 * kIssPP;
  static constexpr int kCopyWarp = kIssWarp + kIssN;        // x (TMA)
  static constexpr int kCodeWarp = kCopyWarp + 1;           // codes (bulk copies)
  static constexpr int kEpiWarp = kCodeWarp + 1;            // 4 epilogue warps
  static constexpr int kThreads = (kEpiWarp + 4) * 32;
  static constexpr int kN = 2 * TOK;                        // B rows: Re x, then Im x
  static constexpr int kAccCols = kN;                       // columns of one accumulator
  static constexpr int kSub = TOK / 16;                     // 16-token sub-blocks of a tile
  static constexpr int kXSub = 2 * TOK * 128;               // x of 64 codes: 2 parts x TOK x 128 B
  static constexpr int kXStage = 2 * kXSub;                 // x stage: 128 codes
  // kind::f16, bf16 A and B (format 1), f32 D, K-major, N = kN, M = 128.
  static constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) |
                                     ((uint32_t)(kN >> 3) << 17) | ((128u >> 4) << 24);
  static constexpr int kOffX = 0;                           // 1024-aligned (swizzle 128 B)
  static constexpr int kOffCodes = kOffX + kXS * kXStage;
  static constexpr int kOffRed = kOffCodes + kCS * kCStage;
  static constexpr int kOffBar = kOffRed + kRed * 4;
  static constexpr int kNumBars = 2 * kXS + 2 * kCS + 2 * kG + 5 + kIssN;
  static constexpr int kOffMisc = kOffBar + kNumBars * 8;
  static constexpr int kSmemBytes = kOffMisc + 64 + 1024;
  static_assert(2 * kIssPP * kAccCols <= kColA, "accumulators");
  static_assert(kSmemBytes > 116 * 1024, "one CTA per SM: it owns all TMEM columns");
  static_assert(kSmemBytes <= 227 * 1024, "shared memory per CTA");
};

constexpr int kMaxGroup = 4;
constexpr int64_t kTwoLaunchMinTokens = 512;   // T = 3 as a T = 2 and a T = 1 launch from here on

struct Args {
  const uint32_t* codes[kMaxGroup];   // linears sharing x (a group), same shape
  const float* scales[kMaxGroup];
  float* y[kMaxGroup];
  int G;            // linears of the group
  unsigned int* status;
  int64_t B, n, out_features, ldy;
  int wpr;          // code words per row (steps of 16 codes)
  int nch;          // 128-code chunks per row (= x stages per tile)
  int row_tiles;    // ceil(n / 16)
  int row_blocks;   // ceil(n / R) per linear
  int tok_tiles;    // ceil(B / TOK)
  int split;        // 2: clusters of two CTAs split each tile's chunks; 1: one CTA per tile
  int accumulate;   // 1: y += the result (the second launch of a two-launch T = 3 layer)
};

// Tile t (token-tile-major, so that CTAs (or CTA pairs) running together share x in L2): token
// tile tb, linear g, row block rb.
__device__ __forceinline__ void tile_coords(const Args& a, int tile, int& g, int& rb, int& tb) {
  const int per_tok = a.G * a.row_blocks;
  tb = tile / per_tok;
  const int rest = tile - tb * per_tok;
  g = rest / a.row_blocks;
  rb = rest - g * a.row_blocks;
}

// Shared-memory descriptor of a K-major operand in the 128-byte swizzle layout: rows of 128 B
// (64 bf16 of K), 8-row groups 1024 B apart; start address advanced by 32 B per 16-element step.
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t addr) {
  return (uint64_t)((addr >> 4) & 0x3FFFu) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
         (1ull << 46) | (2ull << 61);
}

__device__ __forceinline__ void mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                            uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %3, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %4, p;\n}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(accumulate), "r"(idesc)
      : "memory");
}

// bf16 +-1 pairs of one sign plane of a code word: p holds the plane's even-code bits in byte 1
// and odd-code bits in byte 3; register c = (code 2c, code 2c+1), 1 - 2 bit each.
__device__ __forceinline__ void plane_bf16(uint32_t p, uint32_t* r) {
#pragma unroll
  for (int c = 0; c < 8; ++c) r[c] = lop3_and_or(p << (7 - c), 0x80008000u, 0x3F803F80u);
}

// Bounded wait; the first try is the fast path, the abort flag is looked at only after it fails.
__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, volatile int* abort,
                                              unsigned int* status) {
  if (mbar_try_wait(bar, parity)) return true;
  if (*abort) return false;
  if (mbar_wait_timed(bar, parity, kWaitNs)) return true;
  *abort = 1;
  latch_status(status, kStatusTimeout);
  return false;
}
// The same for the two MMA-issuing threads: they spin, so that a group's MMAs follow its A
// stores without a suspended thread's wake-up delay (the issuers are the tensor pipe's feed).
__device__ __forceinline__ bool spin_or_abort(uint64_t* bar, uint32_t parity, volatile int* abort,
                                              unsigned int* status) {
  if (mbar_test_wait(bar, parity)) return true;
  if (*abort) return false;
  if (mbar_wait_spin(bar, parity, kWaitNs)) return true;
  *abort = 1;
  latch_status(status, kStatusTimeout);
  return false;
}

template <int T, int TOK>
__global__ void __launch_bounds__(Cfg<TOK>::kThreads, 1)
    wl_prefill_kernel(const __grid_constant__ Args a, const __grid_constant__ CUtensorMap xre,
                      const __grid_constant__ CUtensorMap xim) {
  using C = Cfg<TOK>;
  constexpr int kIssPP = C::kIssPP, kIssN = C::kIssN, kCopyWarp = C::kCopyWarp;
  constexpr int kXSub = C::kXSub, kXStage = C::kXStage, kOffX = C::kOffX;
  constexpr int kOffCodes = C::kOffCodes, kOffRed = C::kOffRed, kOffBar = C::kOffBar;
  constexpr int kOffMisc = C::kOffMisc;
  constexpr int TM = 2 * T;
  constexpr int R = (T == 1) ? 64 : (T == 2 ? 32 : 16);
  constexpr int RT = R / 16;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = align_smem_1024(smem_raw);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kOffBar);
  uint64_t* xfull = bars;                   // x stage landed            (tx)
  uint64_t* xempty = xfull + kXS;           // x stage consumed          (2 kIssPP issuer commits)
  uint64_t* cfull = xempty + kXS;           // code stage landed         (tx)
  uint64_t* cempty = cfull + kCS;           // code stage read           (8 decoder warps)
  uint64_t* gfull = cempty + kCS;           // group's A stored, x in    (4 warps x 2 pairs)
  uint64_t* gempty = gfull + kG;            // group's A consumed        (2 issuer commits)
  uint64_t* accf = gempty + kG;             // tile accumulators final   (every issuer commits)
  uint64_t* dempty = accf + 1;              // accumulators read out     (4 epilogue warps)
  uint64_t* fin = dempty + 1;               // [issuer] issued MMAs complete (end of kernel)
  uint64_t* ebar = fin + kIssN;             // epilogue warps' barrier (128 threads)
  uint64_t* pready = ebar + 1;              // K split, rank 0: rank 1's sums stored (128)
  uint64_t* pfree = pready + 1;             // K split, rank 1: rank 0 has read them (1)
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + kOffMisc);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kOffMisc + 8);
  float* red = reinterpret_cast<float*>(smem + kOffRed);

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool split = a.split == 2;
  const int rank = split ? (int)cluster_ctarank() : 0;
  const int unit = split ? (int)blockIdx.x >> 1 : (int)blockIdx.x;     // CTA or CTA pair
  const int nunits = split ? (int)gridDim.x >> 1 : (int)gridDim.x;
  const int ntiles = a.G * a.row_blocks * a.tok_tiles;
  const int my_tiles = ntiles > unit ? (ntiles - 1 - unit) / nunits + 1 : 0;
  // this CTA's 128-code chunks of every tile: [c0, c0 + nch)
  const int c0 = (split && rank == 1) ? a.nch / 2 : 0;
  const int nch = split ? (rank == 0 ? a.nch / 2 : a.nch - a.nch / 2) : a.nch;   // x stages
  const int gpt = 2 * nch;            // groups per tile (2 per chunk)

  if (tid == 0) {
    for (int i = 0; i < kXS; ++i) {
      mbar_init(&xfull[i], 1);
      mbar_init(&xempty[i], 2 * kIssPP);
    }
    for (int i = 0; i < kCS; ++i) {
      mbar_init(&cfull[i], 1);
      mbar_init(&cempty[i], 8);
    }
    for (int i = 0; i < kG; ++i) {
      mbar_init(&gfull[i], 8);
      mbar_init(&gempty[i], 2);
    }
    mbar_init(accf, kIssN);
    mbar_init(dempty, 4);
    for (int i = 0; i < kIssN; ++i) mbar_init(&fin[i], 1);
    mbar_init(ebar, 128);
    mbar_init(pready, 128);
    mbar_init(pfree, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(tmem_slot, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  if (split) cluster_arrive_relaxed();   // both ranks' barriers initialised (waited before remote use)
  pdl_launch_dependents();

  if (warp == kCopyWarp) {
    // ---------------- producer of x (TMA), in K order ----------------
    if (lane == 0) {
      prefetch_tensormap(&xre);
      prefetch_tensormap(&xim);
    }
    bool waited = false;
    int xq = 0;   // running stage counter over all tiles of this CTA
    for (int it = 0; it < my_tiles && !__shfl_sync(0xffffffffu, *abort_flag, 0); ++it) {
      const int tile = unit + it * nunits;
      int g, rb, tb;
      tile_coords(a, tile, g, rb, tb);
      bool ok = true;
      for (int xs = c0; xs < c0 + nch; ++xs, ++xq) {
        const int xst = xq % kXS;
        bool okx = true;
        if (lane == 0 && xq >= kXS)
          okx = wait_or_abort(&xempty[xst], ((xq / kXS) - 1) & 1, abort_flag, a.status);
        if (!__shfl_sync(0xffffffffu, okx, 0)) {
          ok = false;
          break;
        }
        if (!waited) {   // x may be written by the previous kernel
          pdl_wait_primary();
          waited = true;
        }
        if (lane == 0) {
          mbar_arrive_expect_tx(&xfull[xst], (uint32_t)kXStage);
          unsigned char* dst = smem + kOffX + xst * kXStage;
          tma_load_2d(dst, &xre, xs * 128, tb * TOK, &xfull[xst]);
          tma_load_2d(dst + kXSub / 2, &xim, xs * 128, tb * TOK, &xfull[xst]);
          tma_load_2d(dst + kXSub, &xre, xs * 128 + 64, tb * TOK, &xfull[xst]);
          tma_load_2d(dst + kXSub + kXSub / 2, &xim, xs * 128 + 64, tb * TOK, &xfull[xst]);
        }
        __syncwarp();
      }
      if (!ok) break;
    }
    // Copies still in flight (after an abort) land before the CTA exits: wait for the last phase
    // of every stage that was filled.
    if (lane == 0)
      for (int q = max(0, xq - kXS); q < xq; ++q)
        (void)mbar_wait_timed(&xfull[q % kXS], (q / kXS) & 1, kWaitNs);
    __syncwarp();
  } else if (warp == C::kCodeWarp) {
    // ---- producer of the codes (bulk copies of whole 16-row tiles, kCChunks chunks a stage):
    // its own warp, since a thread issuing copies blocks on each, and ahead of x (codes are not
    // written by a kernel that lets this one start early, so no griddepcontrol.wait) ----
    int cq = 0;   // running stage counter over all tiles of this CTA
    for (int it = 0; it < my_tiles && !__shfl_sync(0xffffffffu, *abort_flag, 0); ++it) {
      const int tile = unit + it * nunits;
      int g, rb, tb;
      tile_coords(a, tile, g, rb, tb);
      const uint32_t* codes = a.codes[g];
      int ntl = 0;
#pragma unroll
      for (int rt = 0; rt < RT; ++rt) ntl += (rb * RT + rt < a.row_tiles) ? 1 : 0;
      bool ok = true;
      for (int xs = c0; xs < c0 + nch; xs += kCChunks, ++cq) {   // chunks xs .. xs + nc - 1
        const int st = cq % kCS;
        const int nc = min(kCChunks, c0 + nch - xs);
        ok = cq < kCS ||
             lane != 0 || wait_or_abort(&cempty[st], ((cq / kCS) - 1) & 1, abort_flag, a.status);
        if (!__all_sync(0xffffffffu, ok)) {
          ok = false;
          break;
        }
        if (lane == 0) mbar_arrive_expect_tx(&cfull[st], (uint32_t)(TM * ntl * nc * 512));
        __syncwarp();
        const int tm = lane / RT, rt = lane % RT;
        if (lane < TM * RT && rt < ntl) {
          const int64_t t16 = (int64_t)tm * a.row_tiles + rb * RT + rt;
          bulk_load(smem + kOffCodes + st * kCStage + lane * kCChunks * 512,
                    codes + (t16 * a.nch + xs) * 128, (uint32_t)(nc * 512), &cfull[st]);
        }
      }
      if (!ok) break;
    }
    if (lane == 0)
      for (int q = max(0, cq - kCS); q < cq; ++q)
        (void)mbar_wait_timed(&cfull[q % kCS], (q / kCS) & 1, kWaitNs);
    __syncwarp();
  } else if (warp >= kIssWarp && warp < kIssWarp + kIssN) {
    // ---- MMA issuers: warp kIssWarp + kIssPP p + e issues, for sign plane p (sigma, tau), the
    // groups gi = e, e + kIssPP, ... of every tile into its own accumulator ----
    const int ii = warp - kIssWarp, plane = ii / kIssPP, e = ii % kIssPP;
    if (lane == 0) {
      int gbase = 0;   // groups of the earlier tiles
      const uint32_t dcol = tmem + kColD + (uint32_t)(ii * C::kAccCols);
      for (int it = 0; it < my_tiles; ++it, gbase += gpt) {
        if (it > 0 && !spin_or_abort(dempty, (it - 1) & 1, abort_flag, a.status)) break;
        tc_fence_after();
        bool ok = true;
        for (int gi = e; gi < gpt; gi += kIssPP) {
          const int g = gbase + gi;
          const int slot = g % kG;
          const int xst = (it * nch + (gi >> 1)) % kXS;
          if (!spin_or_abort(&gfull[slot], (g / kG) & 1, abort_flag, a.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t xaddr = smem_u32(smem + kOffX + xst * kXStage + (gi & 1) * kXSub);
          const uint32_t acol = tmem + kColA + slot * 64 + plane * 8;
#pragma unroll
          for (int k = 0; k < 4; ++k)   // step k of the group: pair k / 2, step k % 2 of the pair
            mma_bf16_ts(dcol, acol + (k >> 1) * 32 + (k & 1) * 16, smem_desc_sw128(xaddr + k * 32),
                        C::kIdesc, (gi > e || k > 0) ? 1u : 0u);
          mma_commit(&gempty[slot]);
          // this thread's last group of the x stage (groups 2 s, 2 s + 1)
          if (kIssPP == 2 || (gi & 1)) mma_commit(&xempty[xst]);
        }
        if (!ok) break;
        mma_commit(accf);
      }
      // Every MMA this thread issued completes before TMEM is released.
      mma_commit(&fin[ii]);
      (void)mbar_wait_timed(&fin[ii], 0, kWaitNs);
    }
    __syncwarp();
  } else if (warp < kIssWarp) {
    // ---------------- warps 0-7: decode ----------------
    const int set = warp >> 2, quarter = warp & 3, L = quarter * 32 + lane;
    const uint32_t t_lane = tmem + ((uint32_t)(quarter * 32) << 16);
    const int tl = L >> 4, rl = L & 15;   // 16-row tile (tm * RT + rt) and row within it
    const bool relay = warp == 0;         // waits for each x stage before announcing its groups
    int g = 0;                            // running group counter
    int cq0 = 0;                          // code stages of the earlier tiles
    for (int it = 0; it < my_tiles; ++it) {
      bool ok = true;
      // Two groups (the two halves of one x stage) per iteration, so that the waits and the
      // barrier traffic are paid once per pair. Software pipeline: the A stores of a pair are in
      // flight while the next pair is decoded; their barrier arrivals follow the store wait at the
      // next iteration (the relay warp's after the pair's x stage has landed: only the MMAs need
      // x, not the decode).
      int pend = -1, pend_xq = 0;         // first slot and x stage of the pair stored, not announced
      auto announce = [&]() -> bool {
        tmem_wait_st();
        tc_fence_before();
        if (relay) {
          bool okx = true;
          if (lane == 0)
            okx = wait_or_abort(&xfull[pend_xq % kXS], (pend_xq / kXS) & 1, abort_flag, a.status);
          if (!__shfl_sync(0xffffffffu, okx, 0)) return false;
        }
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&gfull[pend]);
          mbar_arrive(&gfull[pend + 1]);
        }
        pend = -1;
        return true;
      };
      for (int gi = 0; gi < gpt; gi += 2, g += 2) {   // gpt, g even: slots g % kG, g % kG + 1
        const int slot = g % kG;
        const int cq = cq0 + gi / kGroupsPerCStage, st = cq % kCS;
        if (gi % kGroupsPerCStage == 0)
          ok = __all_sync(0xffffffffu, wait_or_abort(&cfull[st], (cq / kCS) & 1, abort_flag, a.status));
        if (!ok) break;
        // first word of pair `set` of group gi in the stage; group gi + 1's is 4 words on, in the
        // same 128-code chunk
        const int wi = (gi % kGroupsPerCStage) * 4 + set * 2;
        const unsigned char* cw = smem + kOffCodes + st * kCStage +
                                  (tl * kCChunks + (wi >> 3)) * 512 + rl * 32 + (wi & 7) * 4;
        const uint2 w2a = *reinterpret_cast<const uint2*>(cw);
        const uint2 w2b = *reinterpret_cast<const uint2*>(cw + 16);
        uint32_t r[32];
        plane_bf16(prmt(w2a.x, 0u, 0x1404u), r);        // sigma, first step of the pair
        plane_bf16(prmt(w2a.x, 0u, 0x3424u), r + 8);    // tau
        plane_bf16(prmt(w2a.y, 0u, 0x1404u), r + 16);   // sigma, second step
        plane_bf16(prmt(w2a.y, 0u, 0x3424u), r + 24);   // tau
        if (pend >= 0 && !announce()) {
          ok = false;
          break;
        }
        if (g >= kG)
          ok = __all_sync(0xffffffffu, wait_or_abort(&gempty[slot], ((g / kG) - 1) & 1,
                                                     abort_flag, a.status) &&
                                           wait_or_abort(&gempty[slot + 1], ((g / kG) - 1) & 1,
                                                         abort_flag, a.status));
        if (!ok) break;
        tmem_st32(t_lane + kColA + slot * 64 + set * 32, r);
        plane_bf16(prmt(w2b.x, 0u, 0x1404u), r);
        plane_bf16(prmt(w2b.x, 0u, 0x3424u), r + 8);
        plane_bf16(prmt(w2b.y, 0u, 0x1404u), r + 16);
        plane_bf16(prmt(w2b.y, 0u, 0x3424u), r + 24);
        tmem_st32(t_lane + kColA + (slot + 1) * 64 + set * 32, r);
        __syncwarp();
        if (lane == 0 && ((gi + 1) % kGroupsPerCStage == kGroupsPerCStage - 1 || gi + 1 == gpt - 1))
          mbar_arrive(&cempty[st]);   // this warp's last read of the code stage
        pend = slot;
        pend_xq = it * nch + (gi >> 1);
      }
      if (ok && pend >= 0 && !announce()) ok = false;
      cq0 += (gpt + kGroupsPerCStage - 1) / kGroupsPerCStage;
      if (!ok) break;
    }
  } else {
    // ---------------- the last four warps: epilogue of each tile ----------------
    const int quarter = warp & 3, L = quarter * 32 + lane;
    const uint32_t t_lane = tmem + ((uint32_t)(quarter * 32) << 16);
    const int tm = L / R;
    const bool valid = L < TM * R;
    const int t = tm >> 1, mat = tm & 1;
    uint32_t eph = 0;                     // phases of the epilogue barrier passed
    // Barrier of the 128 epilogue threads with a bounded wait (false: the kernel aborts).
    auto epi_sync = [&]() -> bool {
      mbar_arrive(ebar);
      const bool ok = mbar_wait_timed(ebar, eph & 1, kWaitNs);
      ++eph;
      if (!__all_sync(0xffffffffu, ok)) {
        *abort_flag = 1;
        if (lane == 0) latch_status(a.status, kStatusTimeout);
        return false;
      }
      return true;
    };
    if (split) cluster_wait();   // the peer's barriers are initialised
    for (int it = 0; it < my_tiles; ++it) {
      const int tile = unit + it * nunits;
      int g, rb, tb;
      tile_coords(a, tile, g, rb, tb);
      const float hr = valid ? 0.5f * __ldg(a.scales[g] + (t * 2 + mat) * 2 + 0) : 0.f;
      const float hi = valid ? 0.5f * __ldg(a.scales[g] + (t * 2 + mat) * 2 + 1) : 0.f;
      float* const y = a.y[g];
      if (!__all_sync(0xffffffffu, wait_or_abort(accf, it & 1, abort_flag, a.status))) break;
      tc_fence_after();
      // K split, rank 1: rank 0 has read the previous tile's partials out of this CTA's buffer
      if (split && rank == 1 && it > 0 &&
          !__all_sync(0xffffffffu, mbar_wait_cluster_poll(pfree, (it - 1) & 1, kWaitNs))) {
        *abort_flag = 1;
        if (lane == 0) latch_status(a.status, kStatusTimeout);
        break;
      }
#pragma unroll 1
      for (int sb = 0; sb < C::kSub; ++sb) {   // 16 tokens per sub-block
        // accumulator (plane, e): columns [re of the TOK tokens | im]; the issuers of a plane
        // are added in a fixed order
        float pr[16], pi[16], qr[16], qi[16];
        const uint32_t c0 = t_lane + kColD + sb * 16;
        constexpr uint32_t kTau = (uint32_t)(kIssPP * C::kAccCols);
        tmem_ld16(c0, pr);
        tmem_ld16(c0 + TOK, pi);
        tmem_ld16(c0 + kTau, qr);
        tmem_ld16(c0 + kTau + TOK, qi);
        tmem_wait_ld();
        if constexpr (kIssPP == 2) {
          float v[16];
          tmem_ld16(c0 + C::kAccCols, v);
          tmem_wait_ld();
#pragma unroll
          for (int k = 0; k < 16; ++k) pr[k] += v[k];
          tmem_ld16(c0 + C::kAccCols + TOK, v);
          tmem_wait_ld();
#pragma unroll
          for (int k = 0; k < 16; ++k) pi[k] += v[k];
          tmem_ld16(c0 + kTau + C::kAccCols, v);
          tmem_wait_ld();
#pragma unroll
          for (int k = 0; k < 16; ++k) qr[k] += v[k];
          tmem_ld16(c0 + kTau + C::kAccCols + TOK, v);
          tmem_wait_ld();
#pragma unroll
          for (int k = 0; k < 16; ++k) qi[k] += v[k];
        }
        float* sr = red + sb * (16 * 2 * 128);
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          float Pr = pr[k], Pi = pi[k], Qr = qr[k], Qi = qi[k];
          if (mat) {                 // W multiplies conj(x)
            Pi = -Pi;
            Qi = -Qi;
          }
          sr[(k * 2 + 0) * 128 + L] = valid ? hr * Pr - hi * Pi + hr * Qr + hi * Qi : 0.f;
          sr[(k * 2 + 1) * 128 + L] = valid ? hr * Pi + hi * Pr + hr * Qi - hi * Qr : 0.f;
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(dempty);   // the issuers may start the next tile
      if (!epi_sync()) break;
      // Sum over the stage-matrices, four rows at a time. Item = (sub-block, token k, part) at
      // q = 32 sub-block + 2 k + part, rows 4 rq .. 4 rq + 3 of the row block; thread L takes
      // rq = L % kRQ and q = L / kRQ + kTP i (kTP a divisor of 32), so every item of a thread
      // has the same part, its token is (L / kRQ) / 2 + 16 (i / kIPS) + (kTP / 2) (i % kIPS),
      // and its buffer offset a constant from the thread's first once the loop is unrolled.
      constexpr int kRQ = R / 4;
      constexpr int kTP = 128 / kRQ;
      constexpr int kIPS = 32 / kTP;                // items per sub-block and thread
      constexpr int kPerThread = C::kSub * kIPS;
      const int rq = L % kRQ, tp = L / kRQ;
      const float* red_t = red + tp * 128 + 4 * rq;
      auto stage_sum = [&](int i) -> float4 {
        const float* sr = red_t + (i / kIPS) * (16 * 2 * 128) + (i % kIPS) * (kTP * 128);
        float4 sum = *reinterpret_cast<const float4*>(sr);
#pragma unroll
        for (int m2 = 1; m2 < TM; ++m2) {
          const float4 v = *reinterpret_cast<const float4*>(sr + m2 * R);
          sum.x += v.x;
          sum.y += v.y;
          sum.z += v.z;
          sum.w += v.w;
        }
        return sum;
      };
      if (split && rank == 1) {
        // K split, rank 1: the sums, packed at red[4 (128 i + L)] once every thread has read
        // its inputs, then released to rank 0, which reads them
        float4 part[kPerThread];
#pragma unroll
        for (int i = 0; i < kPerThread; ++i) part[i] = stage_sum(i);
        if (!epi_sync()) break;
#pragma unroll
        for (int i = 0; i < kPerThread; ++i) reinterpret_cast<float4*>(red)[128 * i + L] = part[i];
        mbar_arrive_remote(mapa_shared(smem_u32(pready), 0));
        if (__shfl_sync(0xffffffffu, *abort_flag, 0)) break;
        continue;
      }
      if (split && !__all_sync(0xffffffffu, mbar_wait_cluster_poll(pready, it & 1, kWaitNs))) {
        *abort_flag = 1;
        if (lane == 0) latch_status(a.status, kStatusTimeout);
        break;
      }
      // this CTA's sum, plus (K split) rank 1's, in that order; one 16-byte store per item where
      // the four outputs exist and are 16-byte aligned, else one store per existing output
      const int im = tp & 1;
      const int64_t j = (int64_t)rb * R + 4 * rq;
      const int64_t b0 = (int64_t)tb * TOK + (tp >> 1);
      const int64_t nb = a.B - b0;                  // tokens of y from b0 on
      const int64_t lim = im ? min(a.n, a.out_features - a.n) : a.n;   // rows j < lim exist
      float* const yt = y + b0 * a.ldy + im * a.n + j;
      const bool vec = j + 3 < lim && (a.ldy & 3) == 0 && (reinterpret_cast<uintptr_t>(yt) & 15) == 0;
      const uint32_t peer_red = split ? mapa_shared(smem_u32(red), 1) + 16u * L : 0u;
      constexpr int kBatch = kPerThread < 4 ? kPerThread : 4;   // rank 1's sums loaded together
#pragma unroll
      for (int i0 = 0; i0 < kPerThread; i0 += kBatch) {
        float4 other[kBatch];
        if (split) {
#pragma unroll
          for (int u = 0; u < kBatch; ++u) other[u] = ld_cluster_f32x4(peer_red + 2048u * (i0 + u));
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
          const int i = i0 + u;
          float4 out = stage_sum(i);
          if (split) {
            out.x += other[u].x;
            out.y += other[u].y;
            out.z += other[u].z;
            out.w += other[u].w;
          }
          const int db = 16 * (i / kIPS) + (kTP / 2) * (i % kIPS);
          if (db < nb) {
            float* const yp = yt + db * a.ldy;
            if (vec) {
              if (a.accumulate) {   // y (the first launch's stages) + this launch's, in that order
                const float4 y0 = *reinterpret_cast<const float4*>(yp);
                out.x = y0.x + out.x;
                out.y = y0.y + out.y;
                out.z = y0.z + out.z;
                out.w = y0.w + out.w;
              }
              *reinterpret_cast<float4*>(yp) = out;
            } else {
              const float v[4] = {out.x, out.y, out.z, out.w};
#pragma unroll
              for (int c = 0; c < 4; ++c)
                if (j + c < lim) yp[c] = a.accumulate ? yp[c] + v[c] : v[c];
            }
          }
        }
      }
      if (!epi_sync()) break;
      if (split && L == 0) mbar_arrive_remote(mapa_shared(smem_u32(pfree), 1));
      if (__shfl_sync(0xffffffffu, *abort_flag, 0)) break;
    }
  }

  // K split: neither CTA exits while the other may still arrive on its barriers (every wait
  // above is bounded, so every thread of the pair gets here).
  if (split) {
    if (warp < C::kEpiWarp) cluster_wait();   // the epilogue warps waited the first phase
    cluster_arrive();
    cluster_wait();
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0) tmem_dealloc(tmem, kTmemCols);
}

template <int T, int TOK>
fairy2i_status launch(const Args& a, const CUtensorMap& xre, const CUtensorMap& xim, int grid,
                      cudaStream_t stream) {
  auto kern = wl_prefill_kernel<T, TOK>;
  static std::atomic<uint64_t> smem_set{0};
  if (!smem_attr_once(kern, Cfg<TOK>::kSmemBytes, smem_set)) return FAIRY2I_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(Cfg<TOK>::kThreads);
  cfg.dynamicSmemBytes = Cfg<TOK>::kSmemBytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = (unsigned)a.split;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = a.split == 2 ? 2 : 1;
  if (cudaLaunchKernelEx(&cfg, kern, a, xre, xim) != cudaSuccess) return FAIRY2I_ERR_CUDA;
  return FAIRY2I_OK;
}

// CTA pairs (clusters of two) of the kernel that can be resident at once; 0 if none.
template <int T, int TOK>
int max_pairs() {
  auto kern = wl_prefill_kernel<T, TOK>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           Cfg<TOK>::kSmemBytes) != cudaSuccess)
    return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * 256);
  cfg.blockDim = dim3(Cfg<TOK>::kThreads);
  cfg.dynamicSmemBytes = Cfg<TOK>::kSmemBytes;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
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

inline int max_pairs_t(int T, int tok) {
  switch (T * 2 + (tok == 32 ? 1 : 0)) {
    case 1 * 2: return max_pairs<1, 64>();
    case 2 * 2: return max_pairs<2, 64>();
    case 3 * 2: return max_pairs<3, 64>();
    case 4 * 2: return max_pairs<4, 64>();
    case 1 * 2 + 1: return max_pairs<1, 32>();
    case 2 * 2 + 1: return max_pairs<2, 32>();
    case 3 * 2 + 1: return max_pairs<3, 32>();
    case 4 * 2 + 1: return max_pairs<4, 32>();
  }
  return 0;
}

}  // namespace pfl

namespace {
std::mutex g_pfl_mu;
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
int g_pfl_sms[64];
int g_pfl_pairs[64][4][2];   // [device][T - 1][tok == 32]: resident CTA pairs + 1 (0 = unknown)
}  // namespace

static int pfl_resident_pairs(int dev, int T, int tok) {
  std::lock_guard<std::mutex> lock(g_pfl_mu);
  int& v = g_pfl_pairs[dev][T - 1][tok == 32 ? 1 : 0];
  if (v == 0) v = pfl::max_pairs_t(T, tok) + 1;
  return v - 1;
}

static PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  std::lock_guard<std::mutex> lock(g_pfl_mu);
  if (!g_encode) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return nullptr;
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  return g_encode;
}

// 2-D map over one part of x: `width` bf16 values per token row (zero beyond), rows `ldx` apart,
// B rows; box of 64 values x `tok` tokens, 128-byte swizzle.
static bool encode_x_map(CUtensorMap* map, const void* base, int64_t width, int64_t B,
                         int64_t ldx, int tok) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
  if (!enc || width < 1) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)width, (cuuint64_t)B};
  const cuuint64_t strides[1] = {(cuuint64_t)ldx * 2};
  const cuuint32_t box[2] = {64, (cuuint32_t)tok};
  const cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Handles bf16 x with 16-byte aligned rows (ldx % 8 == 0), m % 8 == 0 and T <= 4, for a group of
// 1..4 linears of the same shape on x (one launch: the tiles of every member); anything else is
// left to the other kernels (*handled = false).
fairy2i_status launch_wl_prefill_group(const void* x, fairy2i_dtype xdt, int64_t B,
                                       int64_t in_features, int64_t ldx, int count,
                                       const uint32_t* const* codes, const float* const* scales,
                                       int64_t n, int64_t m, int64_t out_features, int64_t wpr,
                                       int T, float* const* y, int64_t ldy, cudaStream_t stream,
                                       bool* handled) {
  using namespace pfl;
  *handled = false;
  if (count < 1 || count > kMaxGroup) return FAIRY2I_OK;
  if (xdt != FAIRY2I_BF16 || T > 4 || (reinterpret_cast<uintptr_t>(x) % 16) != 0 ||
      ldx % 8 != 0 || m % 8 != 0 || B > (int64_t(1) << 30) || wpr > (int64_t(1) << 24))
    return FAIRY2I_OK;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return FAIRY2I_ERR_CUDA;
  {
    std::lock_guard<std::mutex> lock(g_pfl_mu);
    if (!g_pfl_sms[dev] &&
        cudaDeviceGetAttribute(&g_pfl_sms[dev], cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return FAIRY2I_ERR_CUDA;
  }
  // token tiles of 32 for batches of at most 32 tokens (two issuing threads per sign plane), else
  // 64
  const int tok = B <= 32 ? 32 : 64;
  CUtensorMap xre, xim;
  const __nv_bfloat16* xb = reinterpret_cast<const __nv_bfloat16*>(x);
  if (!encode_x_map(&xre, xb, m, B, ldx, tok)) return FAIRY2I_OK;
  const bool has_im = in_features > m;
  if (!encode_x_map(&xim, has_im ? xb + m : xb, has_im ? in_features - m : 1, B, ldx, tok))
    return FAIRY2I_OK;
  // One launch over stages [t0, t0 + Tp) of every member; accumulate: y += its result.
  auto run = [&](int Tp, int t0, int accumulate) -> fairy2i_status {
    const int R = Tp == 1 ? 64 : (Tp == 2 ? 32 : 16);
    // words of one stage-matrix's codes ([T][2][row tile][chunk][16 rows][8 words] per member)
    const int64_t sm_words = ((n + 15) / 16) * 16 * wpr;
    Args a;
    for (int g = 0; g < kMaxGroup; ++g) {
      const int gg = g < count ? g : 0;
      a.codes[g] = codes[gg] + (int64_t)t0 * 2 * sm_words;
      a.scales[g] = scales[gg] + t0 * 4;
      a.y[g] = y[gg];
    }
    a.G = count;
    a.accumulate = accumulate;
    a.status = device_status_word();
    a.B = B; a.n = n; a.out_features = out_features; a.ldy = ldy;
    a.wpr = (int)wpr; a.nch = (int)(wpr / 8); a.row_tiles = (int)((n + 15) / 16);
    a.row_blocks = (int)((n + R - 1) / R);
    a.tok_tiles = (int)((B + tok - 1) / tok);
    const int64_t tiles = (int64_t)count * a.row_blocks * a.tok_tiles;
    const int sms = g_pfl_sms[dev];
    int grid = (int)(tiles < sms ? tiles : sms);
    // K split over CTA pairs where it shortens the launch: in full-tile time, a pair finishes a
    // tile in half the time, so ceil(tiles / pairs) / 2 waves against ceil(tiles / SMs); taken
    // when that is at most 0.9 of it (the split adds a hand-over per tile) and every rank has a
    // chunk.
    a.split = 1;
    if (a.nch >= 2) {
      const int pairs = pfl_resident_pairs(dev, Tp, tok);
      if (pairs > 0) {
        const int64_t full_waves = (tiles + sms - 1) / sms;
        const int64_t half_waves = (tiles + pairs - 1) / pairs;
        if (half_waves * 5 <= full_waves * 9) {
          a.split = 2;
          grid = 2 * (int)(tiles < pairs ? tiles : pairs);
        }
      }
    }
    switch (Tp * 2 + (tok == 32 ? 1 : 0)) {
      case 1 * 2: return launch<1, 64>(a, xre, xim, grid, stream);
      case 2 * 2: return launch<2, 64>(a, xre, xim, grid, stream);
      case 3 * 2: return launch<3, 64>(a, xre, xim, grid, stream);
      case 4 * 2: return launch<4, 64>(a, xre, xim, grid, stream);
      case 1 * 2 + 1: return launch<1, 32>(a, xre, xim, grid, stream);
      case 2 * 2 + 1: return launch<2, 32>(a, xre, xim, grid, stream);
      case 3 * 2 + 1: return launch<3, 32>(a, xre, xim, grid, stream);
      case 4 * 2 + 1: return launch<4, 32>(a, xre, xim, grid, stream);
    }
    return FAIRY2I_ERR_INVALID_ARG;
  };
  {
    const int64_t tiles = (int64_t)count * ((n + 15) / 16) * ((B + tok - 1) / tok);
    if (tiles > (int64_t(1) << 30)) return FAIRY2I_OK;
  }
  *handled = true;
  // T = 3 at 16 rows per stage-matrix fills 96 of the 128 accumulator lanes; from
  // kTwoLaunchMinTokens tokens on (where the MMAs, not the per-launch phases, set the time) it
  // runs as stages 0-1 (32 rows each, every lane) and then stage 2 (64 rows) added into y.
  if (T == 3 && B >= kTwoLaunchMinTokens) {
    const fairy2i_status st = run(2, 0, 0);
    if (st != FAIRY2I_OK) return st;
    return run(1, 2, 1);
  }
  return run(T, 0, 0);
}

fairy2i_status launch_wl_prefill(const void* x, fairy2i_dtype xdt, int64_t B, int64_t in_features,
                                 int64_t ldx, const uint32_t* codes, const float* scales,
                                 int64_t n, int64_t m, int64_t out_features, int64_t wpr, int T,
                                 float* y, int64_t ldy, cudaStream_t stream, bool* handled) {
  return launch_wl_prefill_group(x, xdt, B, in_features, ldx, 1, &codes, &scales, n, m,
                                 out_features, wpr, T, &y, ldy, stream, handled);
}

}  // namespace fairy2i
