"""Fairy2i oracle: widely-linear conversion, PhaseQuant, residual quantization, packed codes and
the quantized widely-linear matmul, written out plainly from the paper (arXiv 2512.02901).

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__.smoke() and bench.py's CPU-baseline
legs, never by the product path.

Two arithmetic modes
--------------------
``contract``  the artefacts the library must reproduce bit for bit (U, W, codes, scales). Every
              step that the library performs in float32 is performed here in float32 with one
              IEEE round-to-nearest-even per operation (numpy float32 arithmetic); the scale sums
              are float64 in a fixed summation tree; the scale quotient is one float64 division
              rounded once to float32.
``math``      plain float64 everywhere, no float32 rounding, scales kept as exact float64
              quotients. Used for the mathematical pins (Theorem 1, the residual-norm identity).

Readings where the paper is silent:
* real/imaginary pairing of a real vector is by halves: x~ = [Re x ; Im x]  (Sec. 3.1);
* an odd real dimension is padded by one zero channel appended at its end (Sec. 3.1, Remarks);
* ties of the phase projection are broken the way k = floor(2*theta/pi + 1/2) breaks them, and
  w = 0 maps to +1 (Eq. ifairy-proj, theta = Arg(0) taken as 0);
* an empty code set gives a zero scale (Eq. ifairy-scale divides by its size);
* scales are per tensor, per stage, separately for U and W (Eq. ifairy-scale footnote, Sec. 3.3);
* the residual R^(t) is float32, updated by one correctly rounded add per element;
* the scale sums use the fixed tree of ``fixed_tree_sum``;
* Algorithm 1 is read with the scales of Eq. ifairy-dequant and with the W conj(x) term of
  Eq. widely-linear (see ``wl_matmul``).

Code values: c = k mod 4 for codeword i^k, i.e. 0:+1, 1:+i, 2:-1, 3:-i.
Packed layout (``pack_codes``): see the function docstring.
"""
from __future__ import annotations

import numpy as np

__all__ = [
    "complex_dims", "convert", "realify_lin", "realify_conj", "project", "fixed_tree_sum",
    "axis_scales", "dequant", "residual_quantize", "quantize", "words_per_row", "row_tiles",
    "pack_codes", "unpack_codes", "split_input", "wl_matmul", "wl_matmul_rows", "dense_realified",
    "tolerance_bound", "adjoint_codes", "hermitian_scores", "hermitian_attention", "rmsnorm",
    "silu_mul", "decoder_layer", "quantize_activations_int8", "ste_weight_grad",
    "scale_path_grad",
]

F32 = np.float32
TREE_BLOCK = 256


# --------------------------------------------------------------------------------------------
# Sec. 3.1 -- widely-linear transformation
# --------------------------------------------------------------------------------------------
def complex_dims(rows: int, cols: int) -> tuple[int, int]:
    """(n, m) for a real map R in R^{rows x cols}; an odd dimension gets one zero channel
    appended (Sec. 3.1, Remarks), so n = ceil(rows/2), m = ceil(cols/2)."""
    return (rows + 1) // 2, (cols + 1) // 2


def _padded_blocks(R):
    rows, cols = R.shape
    n, m = complex_dims(rows, cols)
    P = np.zeros((2 * n, 2 * m), dtype=R.dtype)
    P[:rows, :cols] = R
    return P[:n, :m], P[:n, m:], P[n:, :m], P[n:, m:]


def convert(R, mode: str = "contract"):
    """Eq. UW-from-R (Sec. 3.1): Re U = (R11+R22)/2, Im U = (R21-R12)/2, Re W = (R11-R22)/2,
    Im W = (R12+R21)/2 with R partitioned into n x m blocks R_ij.

    contract: R is float32; each block sum/difference is one float32 add, then one float32
    multiply by 0.5 (exact unless the result is subnormal). Returns complex64 U, W.
    math: float64, returns complex128 U, W.
    """
    if mode == "contract":
        R = np.asarray(R, dtype=F32)
        R11, R12, R21, R22 = _padded_blocks(R)
        half = F32(0.5)
        U = np.empty(R11.shape, np.complex64)
        W = np.empty(R11.shape, np.complex64)
        U.real = (R11 + R22) * half
        U.imag = (R21 - R12) * half
        W.real = (R11 - R22) * half
        W.imag = (R12 + R21) * half
        return U, W
    R = np.asarray(R, dtype=np.float64)
    R11, R12, R21, R22 = _padded_blocks(R)
    U = 0.5 * (R11 + R22) + 1j * 0.5 * (R21 - R12)
    W = 0.5 * (R11 - R22) + 1j * 0.5 * (R12 + R21)
    return U, W


def realify_lin(U):
    """Eq. realify-ops: R_lin(U) = [[Re U, -Im U], [Im U, Re U]]."""
    return np.block([[U.real, -U.imag], [U.imag, U.real]])


def realify_conj(W):
    """Eq. realify-ops: R_conj(W) = [[Re W, Im W], [Im W, -Re W]]."""
    return np.block([[W.real, W.imag], [W.imag, -W.real]])


# --------------------------------------------------------------------------------------------
# Sec. 3.2 -- PhaseQuant
# --------------------------------------------------------------------------------------------
def project(re, im):
    """Eq. ifairy-proj: b(w) = argmax_{s in {+-1,+-i}} Re(w conj(s)), as code c (b = i^c).

    Re(w conj(s)) is a, b, -a, -b for s = 1, i, -1, -i (a = Re w, b = Im w), so the winner is
    the larger of |a|, |b| with its sign. On ties the paper's equivalent form
    k = floor(2 Arg(w)/pi + 1/2) decides: Arg = pi/4 -> +i, 3pi/4 -> -1, -3pi/4 -> -i,
    -pi/4 -> +1; and w = 0 -> +1. Comparisons treat -0 as +0.
    """
    a = np.asarray(re)
    b = np.asarray(im)
    aa, ab = np.abs(a), np.abs(b)
    re_wins = np.where(a > 0, 0, 2)
    im_wins = np.where(b > 0, 1, 3)
    # |a| == |b| != 0: the codeword counter-clockwise of the diagonal
    tie = np.where(b > 0, np.where(a > 0, 1, 2), np.where(a < 0, 3, 0))
    tie = np.where(aa == 0, 0, tie)
    c = np.where(aa > ab, re_wins, np.where(ab > aa, im_wins, tie))
    return c.astype(np.uint8)


def fixed_tree_sum(v) -> float:
    """Float64 sum in a fixed order (the paper leaves the order open).

    The values are cut into groups of 256 consecutive entries (the last group zero-padded);
    each group is reduced by halving strides: v[i] += v[i+h] for h = 128, 64, ..., 1, leaving
    the group sum in v[0]. The group sums form the next level and are reduced the same way,
    until a single value is left. An empty input sums to 0.
    """
    v = np.asarray(v, dtype=np.float64).ravel()
    if v.size == 0:
        return 0.0
    while True:
        groups = -(-v.size // TREE_BLOCK)
        g = np.zeros(groups * TREE_BLOCK, dtype=np.float64)
        g[: v.size] = v
        g = g.reshape(groups, TREE_BLOCK)
        h = TREE_BLOCK // 2
        while h >= 1:
            g[:, :h] += g[:, h: 2 * h]
            h //= 2
        v = g[:, 0].copy()
        if v.size == 1:
            return float(v[0])


def axis_scales(re, im, c, mode: str = "contract"):
    """Eq. ifairy-scale: s_re = mean |Re w| over codes in {+-1}, s_im = mean |Im w| over codes
    in {+-i}; per tensor. Sums are float64 over the row-major element order with
    ``fixed_tree_sum``; counts are exact. An empty set gives 0.
    contract: s = float32(S / N) (one float64 division, one rounding). math: s = S / N.
    Returns (s_re, s_im, S_re, S_im, N_re, N_im)."""
    re = np.asarray(re, dtype=np.float64).ravel()
    im = np.asarray(im, dtype=np.float64).ravel()
    c = np.asarray(c).ravel()
    on_re = (c == 0) | (c == 2)
    on_im = ~on_re
    S_re = fixed_tree_sum(np.where(on_re, np.abs(re), 0.0))
    S_im = fixed_tree_sum(np.where(on_im, np.abs(im), 0.0))
    N_re = int(np.count_nonzero(on_re))
    N_im = int(np.count_nonzero(on_im))
    q_re = S_re / N_re if N_re else 0.0
    q_im = S_im / N_im if N_im else 0.0
    if mode == "contract":
        return F32(q_re), F32(q_im), S_re, S_im, N_re, N_im
    return q_re, q_im, S_re, S_im, N_re, N_im


def dequant(c, s_re, s_im):
    """Eq. ifairy-dequant: w^ = s_re b_re + i s_im b_im with b = i^c, as complex128."""
    c = np.asarray(c)
    b_re = np.select([c == 0, c == 2], [1.0, -1.0], 0.0)
    b_im = np.select([c == 1, c == 3], [1.0, -1.0], 0.0)
    return float(s_re) * b_re + 1j * (float(s_im) * b_im)


# --------------------------------------------------------------------------------------------
# Sec. 3.3 -- recursive residual quantization
# --------------------------------------------------------------------------------------------
def residual_quantize(M, T: int, mode: str = "contract"):
    """Sec. 3.3, formal definition: R^(0) = M; for t < T: B^(t) = PhaseQuant(R^(t)) with scales
    s^(t) (Eq. ifairy-scale), W^(t) = s_re B_re + i s_im B_im, R^(t+1) = R^(t) - W^(t).

    contract: R is complex64 and each update is one float32 add per element:
    c=0: re - s_re, c=2: re + s_re, c=1: im - s_im, c=3: im + s_im.
    math: R is complex128 and s are exact float64 quotients.
    Returns codes uint8 [T][n][m], scales [T][2] (s_re, s_im) and the residuals R^(0..T).
    """
    if mode == "contract":
        re = np.array(np.real(M), dtype=F32)
        im = np.array(np.imag(M), dtype=F32)
        sdt = F32
    else:
        re = np.array(np.real(M), dtype=np.float64)
        im = np.array(np.imag(M), dtype=np.float64)
        sdt = np.float64
    codes, scales, residuals = [], [], [(re.copy(), im.copy())]
    for _ in range(T):
        c = project(re, im)
        s_re, s_im = axis_scales(re, im, c, mode)[:2]
        s_re, s_im = sdt(s_re), sdt(s_im)
        re = np.where(c == 0, re - s_re, np.where(c == 2, re + s_re, re)).astype(sdt)
        im = np.where(c == 1, im - s_im, np.where(c == 3, im + s_im, im)).astype(sdt)
        codes.append(c)
        scales.append((s_re, s_im))
        residuals.append((re.copy(), im.copy()))
    return np.array(codes, dtype=np.uint8).reshape((T,) + np.shape(M)), \
        np.array(scales, dtype=sdt).reshape(T, 2), residuals


def quantize(U, W, T: int, mode: str = "contract"):
    """Residual quantization applied independently to U and W (Sec. 3.2 Remark ii, Sec. 3.3).
    Returns codes uint8 [T][2][n][m] (index 1: 0 = U, 1 = W) and scales [T][2][2]
    (index 2: 0 = s_re, 1 = s_im)."""
    cu, su, _ = residual_quantize(U, T, mode)
    cw, sw, _ = residual_quantize(W, T, mode)
    return np.stack([cu, cw], axis=1), np.stack([su, sw], axis=1)


# --------------------------------------------------------------------------------------------
# Sec. 3.4 -- 2-bit storage
# --------------------------------------------------------------------------------------------
def words_per_row(m: int) -> int:
    """32-bit words per packed code row: 16 codes per word, rows padded to 128 codes."""
    return -(-m // 128) * 8


def row_tiles(n: int) -> int:
    """Packed rows come in tiles of 16 (the last one zero-padded)."""
    return -(-n // 16)


def _bit_of_lane(i):
    """Bit of the (Re+Im<0) flag of code i (0..15) inside its word: even codes fill byte 0,
    odd codes byte 1, in order; the (Re-Im<0) flag sits 16 bits higher."""
    return 8 * (i & 1) + (i >> 1)


def pack_codes(codes):
    """2 bits per complex weight (Sec. 3.4, storage).

    Word format: the 16 codes i = 0..15 of a word (code k of a row: word k // 16, i = k % 16)
    each own two bits,
        bit b(i)      = 1 iff c in {2, 3}   (the codeword has Re + Im < 0)
        bit 16 + b(i) = 1 iff c in {1, 2}   (the codeword has Re - Im < 0)
    with b(i) = 8 (i % 2) + i // 2: byte 0 holds the first flag of the even codes, byte 1 of
    the odd codes, bytes 2 and 3 the second flag likewise.
    Buffer order: codes [T][2][n][m] are padded to [T][2][16 R][8 C words] (R = row_tiles(n),
    C = words_per_row(m) / 8; padding codes are 0) and stored as
    uint32 [T][2][R][C][16 rows][8 words]: a 16-row x 128-code block is 512 contiguous bytes.
    Returns a flat uint32 array."""
    codes = np.asarray(codes, dtype=np.uint32)
    T, two, n, m = codes.shape
    wpr = words_per_row(m)
    R = row_tiles(n)
    full = np.zeros((T, two, R * 16, wpr * 16), dtype=np.uint32)
    full[:, :, :n, :m] = codes
    full = full.reshape(T, two, R * 16, wpr, 16)
    neg_sum = ((full == 2) | (full == 3)).astype(np.uint64)
    neg_diff = ((full == 1) | (full == 2)).astype(np.uint64)
    bit = np.array([_bit_of_lane(i) for i in range(16)], dtype=np.uint64)
    words = ((neg_sum << bit) + (neg_diff << (bit + 16))).sum(axis=-1).astype(np.uint32)
    words = words.reshape(T, two, R, 16, wpr // 8, 8).transpose(0, 1, 2, 4, 3, 5)
    return np.ascontiguousarray(words).reshape(-1)


def unpack_codes(words, T: int, n: int, m: int):
    """Inverse of ``pack_codes``: uint8 codes [T][2][n][m]."""
    wpr = words_per_row(m)
    R = row_tiles(n)
    w = np.asarray(words, dtype=np.uint32).reshape(T, 2, R, wpr // 8, 16, 8)
    w = w.transpose(0, 1, 2, 4, 3, 5).reshape(T, 2, R * 16, wpr)
    bit = np.array([_bit_of_lane(i) for i in range(16)], dtype=np.uint32)
    neg_sum = (w[..., None] >> bit) & 1
    neg_diff = (w[..., None] >> (bit + 16)) & 1
    # (neg_sum, neg_diff): (0,0) -> 0, (0,1) -> 1, (1,1) -> 2, (1,0) -> 3
    c = np.where(neg_sum == 0, neg_diff, 3 - neg_diff)
    c = c.reshape(T, 2, R * 16, wpr * 16)
    return c[:, :, :n, :m].astype(np.uint8)


# --------------------------------------------------------------------------------------------
# Eq. widely-linear + Eq. res-sum -- the quantized widely-linear matmul
# --------------------------------------------------------------------------------------------
def split_input(x, m: int):
    """Real activations x~ [B][in_features] -> complex x [B][m], x = x~[:m] + i x~[m:] with a
    zero appended when in_features is odd (Sec. 3.1)."""
    x = np.asarray(x, dtype=np.float64)
    Bt, cols = x.shape
    pad = np.zeros((Bt, 2 * m), dtype=np.float64)
    pad[:, :cols] = x
    return pad[:, :m] + 1j * pad[:, m:]


def wl_matmul_rows(x, codes, scales, rows=None):
    """y[:, rows] of y = sum_t (U^(t) x + W^(t) conj(x)) (Eq. widely-linear with Eq. res-sum),
    U^(t), W^(t) dequantized by Eq. ifairy-dequant from codes [T][2][n][m] and float32 scales
    [T][2][2], in complex128. x is complex [B][m]. Returns complex [B][len(rows)].

    This is the plain definition; Algorithm 1 evaluates the same sum multiplication-free, with
    its scales read as in Eq. ifairy-dequant (s_re on the +-1 codes, s_im on the +-i codes) and
    with the W conj(x) term the widely-linear form requires."""
    codes = np.asarray(codes)
    T, _, n, m = codes.shape
    if rows is None:
        rows = np.arange(n)
    rows = np.asarray(rows)
    y = np.zeros((x.shape[0], rows.size), dtype=np.complex128)
    for t in range(T):
        for M, z in ((0, x), (1, np.conj(x))):
            What = dequant(codes[t, M][rows], scales[t][M][0], scales[t][M][1])
            y += z @ What.T
    return y


def wl_matmul(x, codes, scales, out_features: int):
    """Real-layout wrapper: x~ [B][in_features] -> y~ [B][out_features] = [Re y ; Im y], the
    padded output channel of an odd out_features discarded (Sec. 3.1)."""
    n, m = np.shape(codes)[2], np.shape(codes)[3]
    y = wl_matmul_rows(split_input(x, m), codes, scales)
    return np.concatenate([y.real, y.imag], axis=1)[:, :out_features]


def adjoint_codes(codes):
    """Codes of the adjoint layer, whose real map is R^T (the input gradient of the quantized
    layer, the straight-through backward of Sec. 3.2 / Sec. 3.3 for x).

    From Eq. realify-ops: R_lin(U)^T = R_lin(U^H) and R_conj(W)^T = R_conj(W^T), so the transpose
    of R^ = sum_t R_lin(U^(t)) + R_conj(W^(t)) (Eq. R-sum) is the widely-linear map with
    U' = U^(t)H and W' = W^(t)T, both m x n. With U^ = s_re b_re + i s_im b_im (Eq.
    ifairy-dequant), U^H holds conj(b) = i^(-c) with the same scales: the U codes are transposed
    and conjugated (c -> (4 - c) mod 4), the W codes transposed; the scales do not change.
    codes [T][2][n][m] -> [T][2][m][n]."""
    codes = np.asarray(codes)
    out = np.ascontiguousarray(np.transpose(codes, (0, 1, 3, 2))).astype(np.int64)
    out[:, 0] = (4 - out[:, 0]) % 4
    return out.astype(codes.dtype)


def dense_realified(codes, scales):
    """R^ = sum_t R_lin(U^(t)) + R_conj(W^(t)) (Eq. realify-ops, Eq. R-sum), the dense real map
    that the quantized layer applies to x~ = [Re x ; Im x]."""
    codes = np.asarray(codes)
    T, _, n, m = codes.shape
    Rh = np.zeros((2 * n, 2 * m))
    for t in range(T):
        Rh += realify_lin(dequant(codes[t, 0], *scales[t][0]))
        Rh += realify_conj(dequant(codes[t, 1], *scales[t][1]))
    return Rh


def tolerance_bound(x, scales):
    """Per-token bound on |y| for the element-wise tolerance: ||x~||_1 * sum_t s_t, with
    s_t = max(s_re, s_im) of U plus that of W at stage t. Returns [B]."""
    x = np.asarray(x, dtype=np.float64)
    sc = np.asarray(scales, dtype=np.float64)
    s_sum = float(np.sum(np.max(sc, axis=2)))
    return np.abs(x).sum(axis=1) * s_sum


# --------------------------------------------------------------------------------------------
# Sec. 3.1 (self-attention in widely-linear form) -- Hermitian attention and a decoder layer
# --------------------------------------------------------------------------------------------
def hermitian_scores(q, K, heads: int):
    """Eq. hermitian-score for one query token: S[h, l] = Re(q_h^H k_{l,h}) / sqrt(d_k).

    q complex [n], K complex [L][n]; head h is the complex channels [h dc, (h+1) dc) with
    dc = n / heads, and d_k = 2 dc is the head's real dimension (its stacked vector
    [Re q_h ; Im q_h]). Returns float64 [heads][L]."""
    q = np.asarray(q, dtype=np.complex128)
    K = np.asarray(K, dtype=np.complex128)
    n = q.shape[0]
    dc = n // heads
    qh = q.reshape(heads, dc)
    Kh = K.reshape(K.shape[0], heads, dc)
    return np.real(np.einsum("hc,lhc->hl", np.conj(qh), Kh)) / np.sqrt(2.0 * dc)


def hermitian_attention(q, K, V, heads: int):
    """Attention of one query over L keys/values with Hermitian scores (Eq. hermitian-score):
    softmax over l of S[h, l] per head, then o_h = sum_l p[h, l] v_{l,h}; the weights are real,
    so the real and imaginary parts of v are aggregated separately. Returns complex [n]."""
    S = hermitian_scores(q, K, heads)
    P = np.exp(S - S.max(axis=1, keepdims=True))
    P /= P.sum(axis=1, keepdims=True)
    V = np.asarray(V, dtype=np.complex128)
    L, n = V.shape
    dc = n // heads
    return np.einsum("hl,lhc->hc", P, V.reshape(L, heads, dc)).reshape(n)


def rmsnorm(h, w, eps: float):
    """Root-mean-square normalisation of a real vector (the decoder's norm layers stay real:
    the widely-linear rewrite concerns the linear maps only). h, w [d] -> h w / sqrt(mean h^2 + eps)."""
    h = np.asarray(h, dtype=np.float64)
    return h / np.sqrt(np.mean(h * h) + eps) * np.asarray(w, dtype=np.float64)


def silu_mul(g, u):
    """silu(g) * u, the gated activation of the decoder's MLP (real, elementwise)."""
    g = np.asarray(g, dtype=np.float64)
    return g / (1.0 + np.exp(-g)) * np.asarray(u, dtype=np.float64)


def decoder_layer(h, layer, K_cache, V_cache, heads: int, eps: float = 1e-5):
    """One decoder layer for one token (real layout h [d], d = 2 n), every linear the quantized
    widely-linear map (Eq. widely-linear + Eq. res-sum, dequantized by Eq. ifairy-dequant) and
    attention with Hermitian scores (Eq. hermitian-score):
        x = rmsnorm(h) w_attn; q, k, v = Q x, K x, V x (complex); keys/values = cache + (k, v)
        h1 = h + O [Re a ; Im a],  a = attention(q, keys, values)
        x2 = rmsnorm(h1) w_mlp;  h2 = h1 + Down (silu(Gate x2) * Up x2)
    `layer`: dict of (codes, scales) for q, k, v, o, gate, up, down (out/in features implied by
    the codes' shapes) plus w_attn, w_mlp. K_cache, V_cache complex [L][n] (may be empty).
    Returns h2 (float64 [d]) and the new key and value (complex [n])."""
    def lin(name, x, out_features):
        codes, scales = layer[name]
        return wl_matmul(np.asarray(x, np.float64)[None, :], codes, scales, out_features)[0]
    h = np.asarray(h, dtype=np.float64)
    d = h.shape[0]
    n = d // 2
    x = rmsnorm(h, layer["w_attn"], eps)
    q, k, v = (lin(nm, x, d) for nm in ("q", "k", "v"))
    cq, ck, cv = (t[:n] + 1j * t[n:] for t in (q, k, v))
    Kc = np.concatenate([np.asarray(K_cache, np.complex128).reshape(-1, n), ck[None, :]])
    Vc = np.concatenate([np.asarray(V_cache, np.complex128).reshape(-1, n), cv[None, :]])
    a = hermitian_attention(cq, Kc, Vc, heads)
    h1 = h + lin("o", np.concatenate([a.real, a.imag]), d)
    x2 = rmsnorm(h1, layer["w_mlp"], eps)
    dff = 2 * np.shape(layer["gate"][0])[2]
    m = silu_mul(lin("gate", x2, dff), lin("up", x2, dff))
    h2 = h1 + lin("down", m, d)
    return h2, ck, cv


# --------------------------------------------------------------------------------------------
# Sec. 3.4 (LUT-based optimization for CPU) -- int8 activations
# --------------------------------------------------------------------------------------------
def quantize_activations_int8(x):
    """int8 activations for the table-lookup matmul (the paper names INT8 activations without
    fixing the quantizer; read here as per-token symmetric absmax): delta = max|x~| / 127 as one
    float32 division, xq = round-half-even(x~ / delta) in float32, clamped to [-127, 127]; a zero
    token gives delta = 0 and xq = 0. x [in_features] -> (xq int8, delta float32)."""
    x = np.asarray(x, dtype=F32).ravel()
    mx = F32(np.max(np.abs(x))) if x.size else F32(0)
    delta = F32(mx / F32(127))
    if delta == 0:
        return np.zeros(x.shape, np.int8), delta
    q = np.rint(x / delta).astype(F32)
    return np.clip(q, -127, 127).astype(np.int8), delta


# --------------------------------------------------------------------------------------------
# Sec. 3.2 / 3.3 (QAT) -- gradients of the quantized layer
# --------------------------------------------------------------------------------------------
def ste_weight_grad(x, g, n: int, m: int):
    """Gradient of a loss L with respect to the dequantized pair (U^, W^) of a layer, given the
    layer input x~ [B][in_features] and the output gradient g~ = dL/dy~ [B][out_features] (real
    layouts). From y = U^ x + W^ conj(x) (Eq. widely-linear), with complex gradients written as
    dL/dRe + i dL/dIm: dU = sum_b g_b conj(x_b)^T and dW = sum_b g_b x_b^T (complex [n][m]). Under
    the straight-through estimator (Sec. 3.2 QAT) this is the gradient passed to the masters."""
    z = split_input(x, m)
    gc = split_input(g, n)
    return gc.T @ np.conj(z), gc.T @ z


def scale_path_grad(M, codes_M, scales_M, dM, mode: str = "math"):
    """The part of the master gradient that flows through the per-tensor scales (Eq.
    ifairy-scale) of the T residual stages (Sec. 3.3), codes held fixed (straight-through), for
    one matrix M (complex [n][m], float64) with its codes [T][n][m], scales [T][2] and the
    gradient dM = dL/dM^ of the dequantized matrix (complex [n][m]). The loss is linear in the
    scales: L = sum_t a_t s_re^t + c_t s_im^t with a_t = <Re dM, b_re^t>, c_t = <Im dM, b_im^t>.
    Backward through r^(t+1) = r^(t) - (s_re^t b_re^t + i s_im^t b_im^t), r^(0) = M and
    s_re^t = mean over the +-1 codes of |Re r^(t)| (s_im alike):
        s^_t = (a_t, c_t) - <r^_(t+1), b^t> (real and imaginary parts separately),
        r^_t = r^_(t+1) + s^_re,t sign(Re r^(t)) [c in {+-1}] / N_re + i (same for Im),
    from r^_T = 0. Returns (r^_0 = dL/dM through the scales, complex [n][m], and the total scale
    gradients s^ [T][2]). mode "contract" replays the residuals in float32 exactly as the
    quantizer computes them (the library's replay); "math" in float64."""
    codes_M = np.asarray(codes_M)
    T = codes_M.shape[0]
    if mode == "contract":
        # the quantizer's own float32 residuals (one rounding per update)
        re = np.array(np.real(M), dtype=F32)
        im = np.array(np.imag(M), dtype=F32)
        res = [re.astype(np.float64) + 1j * im.astype(np.float64)]
        for t in range(T):
            c = codes_M[t]
            s_re, s_im = F32(scales_M[t][0]), F32(scales_M[t][1])
            re = np.where(c == 0, re - s_re, np.where(c == 2, re + s_re, re)).astype(F32)
            im = np.where(c == 1, im - s_im, np.where(c == 3, im + s_im, im)).astype(F32)
            res.append(re.astype(np.float64) + 1j * im.astype(np.float64))
        M = res[0]
    else:
        M = np.asarray(M, np.complex128)
        res = [M.copy()]
        for t in range(T):
            w = dequant(codes_M[t], scales_M[t][0], scales_M[t][1])
            res.append(res[-1] - w)
    dM = np.asarray(dM, np.complex128)
    rhat = np.zeros_like(M)
    shat = np.zeros((T, 2))
    for t in range(T - 1, -1, -1):
        c = codes_M[t]
        b_re = np.select([c == 0, c == 2], [1.0, -1.0], 0.0)
        b_im = np.select([c == 1, c == 3], [1.0, -1.0], 0.0)
        on_re = (c == 0) | (c == 2)
        on_im = ~on_re
        sre = float(np.sum(dM.real * b_re)) - float(np.sum(rhat.real * b_re))
        sim = float(np.sum(dM.imag * b_im)) - float(np.sum(rhat.imag * b_im))
        shat[t] = (sre, sim)
        r = res[t]
        n_re, n_im = int(on_re.sum()), int(on_im.sum())
        add_re = np.where(on_re, np.sign(r.real) * sre / n_re, 0.0) if n_re else 0.0
        add_im = np.where(on_im, np.sign(r.imag) * sim / n_im, 0.0) if n_im else 0.0
        rhat = rhat + add_re + 1j * add_im
    return rhat, shat
