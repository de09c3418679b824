// Codes of the adjoint layer (the input gradient of the quantized layer, R^T). From the
// realification operators (Eq. realify-ops), R_lin(U)^T = R_lin(U^H) and R_conj(W)^T =
// R_conj(W^T): the adjoint is the widely-linear layer with U' = U^H and W' = W^T, i.e. the code
// matrices transposed, the U codes conjugated (codeword i^c -> i^-c, c -> (4 - c) mod 4), and
// the scales unchanged (Eq. ifairy-dequant). Any matmul path then runs the backward.
//
// One CTA per (stage-matrix, 128-code chunk of the source rows, 128-row block of the source):
// the 8 source row tiles x 128 codes are unpacked into shared memory as one byte per code, then
// packed again as 8 output row tiles (the source codes) x 128 codes (the source rows).
#include <cuda_runtime.h>

#include "common.cuh"

namespace fairy2i {

namespace {

// Bit of the first flag of code i (0..15) in its word: even codes fill byte 0, odd codes byte 1.
__device__ __forceinline__ int flag_bit(int i) { return 8 * (i & 1) + (i >> 1); }

__global__ void __launch_bounds__(256) codes_adjoint_kernel(const uint32_t* __restrict__ src,
                                                            uint32_t* __restrict__ dst, int Rn,
                                                            int Cm, int Rm, int Cn) {
  __shared__ uint8_t S[128][132];   // [source row in the block][source code in the chunk]
  const int c = blockIdx.x;         // source chunk = output row tiles 8 c .. 8 c + 7
  const int rb = blockIdx.y;        // source rows 128 rb .. = output chunk rb
  const int tm = blockIdx.z;        // stage-matrix t * 2 + (0: U, 1: W)
  const bool conj = (tm & 1) == 0;
  for (int q = threadIdx.x; q < 8 * 16 * 8; q += blockDim.x) {
    const int w = q & 7, row = (q >> 3) & 15, tile = q >> 7;
    const int rt = rb * 8 + tile;
    const uint32_t word =
        rt < Rn ? __ldg(src + (((int64_t)tm * Rn + rt) * Cm + c) * 128 + row * 8 + w) : 0u;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int b = flag_bit(i);
      const uint32_t neg_sum = (word >> b) & 1u, neg_diff = (word >> (16 + b)) & 1u;
      uint32_t code = neg_sum ? 3u - neg_diff : neg_diff;   // (0,0) +1, (0,1) +i, (1,1) -1, (1,0) -i
      if (conj) code = (4u - code) & 3u;
      S[tile * 16 + row][w * 16 + i] = (uint8_t)code;
    }
  }
  __syncthreads();
  for (int q = threadIdx.x; q < 128 * 8; q += blockDim.x) {
    const int k = q & 127, w = q >> 7;   // output row k of the chunk, output word w
    const int ot = c * 8 + (k >> 4);
    if (ot >= Rm) continue;
    uint32_t word = 0;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const uint32_t code = S[w * 16 + i][k];
      const int b = flag_bit(i);
      word |= ((code >> 1) & 1u) << b;                                   // c in {2, 3}
      word |= (uint32_t)((code == 1u) | (code == 2u)) << (16 + b);       // c in {1, 2}
    }
    dst[(((int64_t)tm * Rm + ot) * Cn + rb) * 128 + (k & 15) * 8 + w] = word;
  }
}

}  // namespace

fairy2i_status launch_codes_adjoint(const uint32_t* codes, int64_t n, int64_t m, int T,
                                    uint32_t* codes_adj, cudaStream_t stream) {
  const int64_t Rn = (n + 15) / 16, Cm = (m + 127) / 128, Rm = (m + 15) / 16, Cn = (n + 127) / 128;
  if (Cn > 65535 || Cm > (int64_t(1) << 30)) return FAIRY2I_ERR_SHAPE;
  codes_adjoint_kernel<<<dim3((unsigned)Cm, (unsigned)Cn, (unsigned)(2 * T)), 256, 0, stream>>>(
      codes, codes_adj, (int)Rn, (int)Cm, (int)Rm, (int)Cn);
  return cudaGetLastError() == cudaSuccess ? FAIRY2I_OK : FAIRY2I_ERR_CUDA;
}

}  // namespace fairy2i
