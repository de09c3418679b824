// Host (CPU) form of the quantized widely-linear matmul by look-up tables (Sec. 3.4,
// LUT-based optimization for CPU): four 2-bit complex codes form one 8-bit index into a table
// of partial sums precomputed from int8 activations, so the inner loop is a table fetch and an
// integer add per four codes. Portable C++ (no vector intrinsics): it runs on the host cores of
// any machine that loads the library, the Arm cores next to the GPU included.
//
// Index. A packed code word (16 codes, code i at bit b(i) = 8 (i % 2) + i / 2 of the "Re+Im < 0"
// half and 16 + b(i) of the "Re-Im < 0" half) holds four groups: group g (0..3) takes nibble
// g % 2 of byte g / 2 (first flags) and the same nibble of byte 2 + g / 2 (second flags), i.e.
// codes {2 j + (g / 2) + 8 (g % 2) : j = 0..3} -> index = first flags | second flags << 4,
// flag bit j belonging to code 2 j + (g / 2) + 8 (g % 2).
//
// Table of one group (four complex inputs z_0..z_3, int8 parts): for every index, the exact
// integer sums P = sum over the codes in {+1, -1} of b_re z and Q = sum over the codes in
// {+i, -i} of b_im z (complex, int16). For U, w z summed over the group is s_re P + i s_im Q; for
// W the inputs are conj(z), and since b_re, b_im are real the sums are conj(P), conj(Q): one
// table serves both matrices of every stage.
#include <stdint.h>
#include <string.h>

#include <algorithm>
#include <cmath>
#include <thread>
#include <vector>

#include "fairy2i.h"

namespace fairy2i {
namespace {

struct Entry {   // one table entry: P and Q
  int16_t pr, pi, qr, qi;
};

// Builds the 256-entry table of one group from four complex int8 inputs: each entry is the sum of
// its four codes' contributions (eight integer adds), built once per token and group and then
// read by every row.
void build_table(const int8_t* zr, const int8_t* zi, Entry* tab) {
  // contribution of code j for its two flag bits (first, second): (0,0) +1, (0,1) +i,
  // (1,1) -1, (1,0) -i (the packed format's meaning of the two flags)
  for (int idx = 0; idx < 256; ++idx) {
    int pr = 0, pi = 0, qr = 0, qi = 0;
    for (int j = 0; j < 4; ++j) {
      const int f1 = (idx >> j) & 1, f2 = (idx >> (4 + j)) & 1;
      if (f1 == f2) {           // +1 or -1: the real-axis set
        const int sg = f1 ? -1 : 1;
        pr += sg * zr[j];
        pi += sg * zi[j];
      } else {                  // +i (f2) or -i (f1): the imaginary-axis set
        const int sg = f1 ? -1 : 1;
        qr += sg * zr[j];
        qi += sg * zi[j];
      }
    }
    tab[idx] = Entry{(int16_t)pr, (int16_t)pi, (int16_t)qr, (int16_t)qi};
  }
}

}  // namespace
}  // namespace fairy2i

using namespace fairy2i;

extern "C" {

fairy2i_status fairy2i_lut_quantize_x(const float* x, int64_t in_features, int8_t* xq,
                                      float* scale) {
  if (!x || !xq || !scale || in_features < 1) return FAIRY2I_ERR_INVALID_ARG;
  float mx = 0.f;
  for (int64_t i = 0; i < in_features; ++i) {
    const float a = x[i] < 0.f ? -x[i] : x[i];
    if (!(a <= 3.4e38f)) return FAIRY2I_ERR_INVALID_ARG;   // non-finite input
    mx = std::max(mx, a);
  }
  const float delta = mx / 127.0f;
  *scale = delta;
  for (int64_t i = 0; i < in_features; ++i) {
    float q = 0.f;
    if (delta > 0.f) q = nearbyintf(x[i] / delta);          // round half to even
    q = std::min(127.f, std::max(-127.f, q));
    xq[i] = (int8_t)q;
  }
  return FAIRY2I_OK;
}

size_t fairy2i_lut_workspace_bytes(int64_t in_features) {
  if (in_features < 1) return 0;
  const int64_t m = (in_features + 1) / 2;
  const int64_t words = (m + 127) / 128 * 8;
  return (size_t)words * 4 * 256 * sizeof(Entry) + 2 * (size_t)words * 16;
}

fairy2i_status fairy2i_lut_matmul(const int8_t* xq, float x_scale, int64_t in_features,
                                  const uint32_t* codes, const float* scales,
                                  int64_t out_features, int T, float* y, void* workspace,
                                  size_t workspace_bytes, int nthreads) {
  if (!xq || !codes || !scales || !y || in_features < 1 || out_features < 1 || T < 1 ||
      T > FAIRY2I_MAX_STAGES || nthreads < 1 || nthreads > 1024)
    return FAIRY2I_ERR_INVALID_ARG;
  if (!workspace || workspace_bytes < fairy2i_lut_workspace_bytes(in_features))
    return FAIRY2I_ERR_WORKSPACE;
  const int64_t n = (out_features + 1) / 2, m = (in_features + 1) / 2;
  const int64_t wpr = (m + 127) / 128 * 8;          // words per packed row
  const int64_t rtiles = (n + 15) / 16;
  Entry* tabs = static_cast<Entry*>(workspace);      // [word][group][256]
  int8_t* zr = reinterpret_cast<int8_t*>(tabs + wpr * 4 * 256);   // complex inputs, padded
  int8_t* zi = zr + wpr * 16;
  for (int64_t k = 0; k < wpr * 16; ++k) {
    zr[k] = k < m ? xq[k] : 0;
    zi[k] = (k < m && m + k < in_features) ? xq[m + k] : 0;
  }
  // Tables of every group (the words of a row cover codes 16 w .. 16 w + 15).
  auto build = [&](int64_t w0, int64_t w1) {
    for (int64_t w = w0; w < w1; ++w)
      for (int g = 0; g < 4; ++g) {
        int8_t r4[4], i4[4];
        for (int j = 0; j < 4; ++j) {
          const int64_t k = 16 * w + 2 * j + (g / 2) + 8 * (g % 2);
          r4[j] = zr[k];
          i4[j] = zi[k];
        }
        build_table(r4, i4, tabs + (w * 4 + g) * 256);
      }
  };
  // Rows: per (stage, matrix) the integer sums P, Q over the row's groups, then
  // y_j = delta sum_t [s_re P + i s_im Q] (U) + [s_re conj(P) + i s_im conj(Q)] (W).
  auto rows = [&](int64_t j0, int64_t j1) {
    for (int64_t j = j0; j < j1; ++j) {
      const int64_t rt = j / 16, rr = j % 16;
      double yre = 0.0, yim = 0.0;
      for (int t = 0; t < T; ++t)
        for (int M = 0; M < 2; ++M) {
          const uint32_t* base = codes + ((int64_t)(t * 2 + M) * rtiles + rt) * wpr * 16;
          int64_t pr = 0, pi = 0, qr = 0, qi = 0;
          for (int64_t w = 0; w < wpr; ++w) {
            // block layout [chunk][16 rows][8 words]
            const uint32_t cw = base[(w / 8) * 128 + rr * 8 + (w % 8)];
            const Entry* tw = tabs + w * 4 * 256;
            const Entry& e0 = tw[(cw & 0xFu) | ((cw >> 12) & 0xF0u)];
            const Entry& e1 = tw[256 + (((cw >> 4) & 0xFu) | ((cw >> 16) & 0xF0u))];
            const Entry& e2 = tw[512 + (((cw >> 8) & 0xFu) | ((cw >> 20) & 0xF0u))];
            const Entry& e3 = tw[768 + (((cw >> 12) & 0xFu) | ((cw >> 24) & 0xF0u))];
            pr += e0.pr + e1.pr + e2.pr + e3.pr;
            pi += e0.pi + e1.pi + e2.pi + e3.pi;
            qr += e0.qr + e1.qr + e2.qr + e3.qr;
            qi += e0.qi + e1.qi + e2.qi + e3.qi;
          }
          const double s_re = scales[(t * 2 + M) * 2], s_im = scales[(t * 2 + M) * 2 + 1];
          const double sg = M ? -1.0 : 1.0;   // W: conj(P), conj(Q)
          // s_re P + i s_im Q with P, Q conjugated for W
          yre += s_re * (double)pr - s_im * sg * (double)qi;
          yim += s_re * sg * (double)pi + s_im * (double)qr;
        }
      y[j] = (float)(x_scale * yre);
      if (n + j < out_features) y[n + j] = (float)(x_scale * yim);
    }
  };
  const int nt = (int)std::min<int64_t>(nthreads, std::max<int64_t>(1, n / 16));
  if (nt == 1) {
    build(0, wpr);
    rows(0, n);
    return FAIRY2I_OK;
  }
  std::vector<std::thread> pool;
  for (int i = 0; i < nt; ++i)
    pool.emplace_back(build, wpr * i / nt, wpr * (i + 1) / nt);
  for (auto& th : pool) th.join();
  pool.clear();
  for (int i = 0; i < nt; ++i) pool.emplace_back(rows, n * i / nt, n * (i + 1) / nt);
  for (auto& th : pool) th.join();
  return FAIRY2I_OK;
}

}  // extern "C"
