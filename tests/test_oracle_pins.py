"""Pins of the CPU oracle to what the paper and the mathematics fix (no GPU needed).

Each test checks the oracle against something other than itself: Theorem 1 evaluated with
complex arithmetic, closed forms, hand-derived values, brute force over the four codewords,
an exact summation, and the residual-norm identity that follows from Eq. ifairy-scale.
"""
import math
import os

import numpy as np
import pytest

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
rng = np.random.default_rng(12345)

SHAPES = [(2, 2), (6, 8), (7, 9), (5, 4), (33, 17), (64, 130), (1, 3)]


def _real_map_from_complex(U, W):
    """Build R column by column from the complex map x -> U x + W conj(x) applied to the real
    basis: Re-part unit e_k gives column k, Im-part unit i e_k gives column m + k."""
    n, m = U.shape
    R = np.zeros((2 * n, 2 * m))
    for k in range(m):
        y = U[:, k] + W[:, k]                      # x = e_k
        R[:n, k], R[n:, k] = y.real, y.imag
        y = 1j * U[:, k] - 1j * W[:, k]            # x = i e_k, conj(x) = -i e_k
        R[:n, m + k], R[n:, m + k] = y.real, y.imag
    return R


# ---------------------------------------------------------------- Sec. 3.1, Theorem 1
@pytest.mark.parametrize("rows,cols", SHAPES)
def test_theorem1_exact_equivalence(rows, cols):
    R = rng.standard_normal((rows, cols))
    U, W = O.convert(R, mode="math")
    n, m = O.complex_dims(rows, cols)
    assert U.shape == (n, m) and W.shape == (n, m)
    for _ in range(3):
        xt = rng.standard_normal(cols)
        yt = R @ xt
        x = O.split_input(xt[None, :], m)[0]
        y = U @ x + W @ np.conj(x)
        y_real = np.concatenate([y.real, y.imag])
        # the padded output channel of an odd real dimension is discarded
        assert np.max(np.abs(y_real[:rows] - yt)) <= 1e-12 * max(1.0, np.abs(yt).max())
        if rows % 2:
            assert abs(y_real[rows]) <= 1e-12 * max(1.0, np.abs(yt).max())


@pytest.mark.parametrize("n,m", [(3, 5), (8, 8), (1, 1)])
def test_theorem1_uniqueness_inverse(n, m):
    """convert inverts the map (U, W) -> R, where R is built by probing the complex map."""
    U = rng.standard_normal((n, m)) + 1j * rng.standard_normal((n, m))
    W = rng.standard_normal((n, m)) + 1j * rng.standard_normal((n, m))
    R = _real_map_from_complex(U, W)
    U2, W2 = O.convert(R, mode="math")
    assert np.max(np.abs(U2 - U)) < 1e-14 and np.max(np.abs(W2 - W)) < 1e-14


def test_realify_operators_act_like_complex_maps():
    """Eq. realify-eval: R_lin(U) [Re x; Im x] = [Re Ux; Im Ux], R_conj(W) likewise for W conj(x)."""
    n, m = 5, 7
    U = rng.standard_normal((n, m)) + 1j * rng.standard_normal((n, m))
    x = rng.standard_normal(m) + 1j * rng.standard_normal(m)
    xt = np.concatenate([x.real, x.imag])
    a = O.realify_lin(U) @ xt
    b = U @ x
    assert np.allclose(a, np.concatenate([b.real, b.imag]), atol=1e-13, rtol=0)
    a = O.realify_conj(U) @ xt
    b = U @ np.conj(x)
    assert np.allclose(a, np.concatenate([b.real, b.imag]), atol=1e-13, rtol=0)


@pytest.mark.parametrize("rows,cols", [(8, 8), (7, 9), (64, 130)])
def test_R_sum_round_trip(rows, cols):
    """Eq. R-sum: R = R_lin(U) + R_conj(W) for the U, W of Eq. UW-from-R (padded R)."""
    R = rng.standard_normal((rows, cols))
    U, W = O.convert(R, mode="math")
    n, m = U.shape
    P = np.zeros((2 * n, 2 * m))
    P[:rows, :cols] = R
    assert np.max(np.abs(O.realify_lin(U) + O.realify_conj(W) - P)) <= 1e-15 * np.abs(R).max() * 4


def test_convert_special_cases():
    m = 6
    U, W = O.convert(np.eye(2 * m), mode="math")                      # identity: y = x
    assert np.array_equal(U, np.eye(m)) and not np.any(W)
    conj = np.diag(np.r_[np.ones(m), -np.ones(m)])                    # y = conj(x)
    U, W = O.convert(conj, mode="math")
    assert not np.any(U) and np.array_equal(W, np.eye(m))
    C = rng.standard_normal((4, m)) + 1j * rng.standard_normal((4, m))
    lin = np.block([[C.real, -C.imag], [C.imag, C.real]])            # y = C x (C-linear)
    U, W = O.convert(lin, mode="math")
    assert np.allclose(U, C, atol=1e-15) and np.max(np.abs(W)) < 1e-15
    anti = np.block([[C.real, C.imag], [C.imag, -C.real]])           # y = C conj(x)
    U, W = O.convert(anti, mode="math")
    assert np.max(np.abs(U)) < 1e-15 and np.allclose(W, C, atol=1e-15)


def test_convert_contract_is_single_rounding():
    R = rng.standard_normal((40, 34)).astype(np.float32)
    U32, W32 = O.convert(R, mode="contract")
    U64, W64 = O.convert(R.astype(np.float64), mode="math")
    # (a+b)/2 of float32 a, b is exact in float64; float32 add then *0.5 rounds it once
    assert np.array_equal(U32, U64.astype(np.complex64))
    assert np.array_equal(W32, W64.astype(np.complex64))
    assert U32.dtype == np.complex64


# ---------------------------------------------------------------- Sec. 3.2, Eq. ifairy-proj
CODEWORDS = np.array([1, 1j, -1, -1j])


def test_projection_is_argmax_brute_force():
    w = (rng.standard_normal(20000) + 1j * rng.standard_normal(20000)).astype(np.complex64)
    scores = np.real(w.astype(np.complex128)[:, None] * np.conj(CODEWORDS)[None, :])
    best = np.argmax(scores, axis=1)
    top2 = np.sort(scores, axis=1)[:, -2:]
    unique = top2[:, 1] > top2[:, 0]
    c = O.project(w.real, w.imag)
    assert unique.all()
    assert np.array_equal(c, best)


def _k_formula(a, b):
    theta = math.atan2(b, a)
    return math.floor(2 * theta / math.pi + 0.5) % 4


@pytest.mark.parametrize("a,b", [(1, 1), (-1, 1), (-1, -1), (1, -1), (2.5, 2.5), (-3, 3),
                                 (1, 0), (-1, 0), (0, 1), (0, -1), (0.3, 0.1), (-0.2, 0.7)])
def test_projection_ties_follow_floor_formula(a, b):
    """Ties |Re w| = |Im w| are decided as k = floor(2 Arg(w)/pi + 1/2) decides them."""
    assert int(O.project(np.float32(a), np.float32(b))) == _k_formula(a, b)


def test_projection_zero_and_signed_zero():
    z, nz = np.float32(0.0), np.float32(-0.0)
    for a, b in [(z, z), (nz, z), (z, nz), (nz, nz)]:
        assert int(O.project(a, b)) == 0            # Arg(0) taken as 0 -> +1
    assert int(O.project(nz, np.float32(2))) == 1
    assert int(O.project(np.float32(2), nz)) == 0
    assert int(O.project(nz, np.float32(-2))) == 3
    assert int(O.project(np.float32(-2), nz)) == 2


def test_projection_matches_floor_formula_away_from_ties():
    a = rng.standard_normal(5000)
    b = rng.standard_normal(5000)
    ok = np.abs(np.abs(a) - np.abs(b)) > 1e-9
    k = np.array([_k_formula(x, y) for x, y in zip(a, b)])
    assert np.array_equal(O.project(a, b)[ok], k[ok])


def test_fig2_worked_example():
    rows = [l.split() for l in open(os.path.join(GOLDEN, "fig2_projection.txt"))
            if l.strip() and not l.startswith("#")]
    for deg, mag, code in rows:
        th = math.radians(float(deg))
        w = float(mag) * complex(math.cos(th), math.sin(th))
        assert int(O.project(np.float32(w.real), np.float32(w.imag))) == int(code)


# ---------------------------------------------------------------- fixed summation tree
def test_tree_sum_exact_on_exactly_summable_values():
    for size in [0, 1, 2, 255, 256, 257, 65536, 65537, 100003]:
        v = rng.integers(0, 1 << 20, size).astype(np.float64) * 2.0 ** -12
        assert O.fixed_tree_sum(v) == math.fsum(v)


def test_tree_sum_order_hand_derived():
    """[2^53, 1 x 255]: stride-halving pairs (i, i+h) give 2^53 + (2+4+...+128) = 2^53 + 254
    (each partial is exact); summing left to right would give 2^53, fsum 2^53 + 256."""
    v = np.ones(256)
    v[0] = 2.0 ** 53
    assert O.fixed_tree_sum(v) == 2.0 ** 53 + 254
    assert math.fsum(v) == 2.0 ** 53 + 256
    # second level: the same tree over the group sums
    v2 = np.zeros(512)
    v2[0] = 2.0 ** 53
    v2[256] = 1.0
    v2[257] = 1.0
    assert O.fixed_tree_sum(v2) == 2.0 ** 53 + 2


# ---------------------------------------------------------------- Eq. ifairy-scale
def test_scales_hand_example():
    w = np.array([1 + 0.25j, -3 + 1j, 0.5 + 2j, 0.125 - 0.5j], dtype=np.complex64)
    c = O.project(w.real, w.imag)
    assert list(c) == [0, 2, 1, 3]
    s_re, s_im, S_re, S_im, N_re, N_im = O.axis_scales(w.real, w.imag, c)
    assert (N_re, N_im) == (2, 2)
    assert s_re == np.float32(2.0) and s_im == np.float32(1.25)


def test_scales_empty_set_is_zero():
    w = np.array([0.5j, -2j, 1j], dtype=np.complex64)
    c = O.project(w.real, w.imag)
    s_re, s_im = O.axis_scales(w.real, w.imag, c)[:2]
    assert s_re == 0.0 and s_im == np.float32(3.5 / 3)


def test_scales_agree_with_exact_mean():
    w = (0.02 * rng.standard_normal(70001) + 0.02j * rng.standard_normal(70001)).astype(np.complex64)
    c = O.project(w.real, w.imag)
    s_re, s_im = O.axis_scales(w.real, w.imag, c)[:2]
    on_re = (c == 0) | (c == 2)
    e_re = np.float32(math.fsum(np.abs(w.real[on_re]).astype(np.float64)) / on_re.sum())
    e_im = np.float32(math.fsum(np.abs(w.imag[~on_re]).astype(np.float64)) / (~on_re).sum())
    assert abs(int(s_re.view(np.int32)) - int(e_re.view(np.int32))) <= 1
    assert abs(int(s_im.view(np.int32)) - int(e_im.view(np.int32))) <= 1


# ---------------------------------------------------------------- Sec. 3.3, residual stages
def _fro2(re, im):
    return float(np.sum(np.asarray(re, np.float64) ** 2) + np.sum(np.asarray(im, np.float64) ** 2))


@pytest.mark.parametrize("shape", [(17, 33), (128, 128), (3, 1)])
def test_residual_norm_identity_math_mode(shape):
    """On the +-1 set (a - s sgn a)^2 = (|a| - s)^2 and sum |a| = N s, hence
    ||R^(t+1)||^2 = ||R^(t)||^2 - N_re s_re^2 - N_im s_im^2 exactly (math mode)."""
    M = rng.standard_normal(shape) + 1j * rng.standard_normal(shape)
    codes, scales, res = O.residual_quantize(M, 4, mode="math")
    for t in range(4):
        c = codes[t]
        N_re = int(np.count_nonzero((c == 0) | (c == 2)))
        N_im = c.size - N_re
        before = _fro2(*res[t])
        after = _fro2(*res[t + 1])
        expect = before - N_re * scales[t][0] ** 2 - N_im * scales[t][1] ** 2
        assert abs(after - expect) <= 1e-12 * before
        assert after <= before


def test_residual_monotone_contract_mode():
    M = (0.02 * rng.standard_normal((96, 80)) + 0.02j * rng.standard_normal((96, 80))).astype(np.complex64)
    _, _, res = O.residual_quantize(M, 5, mode="contract")
    norms = [_fro2(*r) for r in res]
    assert all(b <= a for a, b in zip(norms, norms[1:]))
    assert norms[1] < 0.5 * norms[0]


def test_T1_reduces_to_phasequant():
    M = (rng.standard_normal((31, 47)) + 1j * rng.standard_normal((31, 47))).astype(np.complex64)
    c1, s1, _ = O.residual_quantize(M, 1)
    c3, s3, _ = O.residual_quantize(M, 3)
    assert np.array_equal(c1[0], c3[0]) and np.array_equal(s1[0], s3[0])
    assert np.array_equal(c1[0], O.project(M.real, M.imag))


def test_single_weight_closed_form():
    """One weight at 60 degrees: stage 0 picks +i with s_im = Im w, leaving the residual
    (Re w, 0); stage 1 picks +1 with s_re = Re w, leaving 0."""
    w = np.array([[np.complex64(0.5 + 0.8660254j)]])
    codes, scales, res = O.residual_quantize(w, 2)
    assert codes[0, 0, 0] == 1 and scales[0][1] == np.float32(0.8660254)
    assert res[1][1][0, 0] == 0.0 and res[1][0][0, 0] == np.float32(0.5)
    assert codes[1, 0, 0] == 0 and scales[1][0] == np.float32(0.5) and res[2][0][0, 0] == 0.0


# ---------------------------------------------------------------- Sec. 3.4, storage
def test_packed_layout_hand_word():
    c = np.zeros((1, 2, 17, 140), dtype=np.uint8)
    c[0, 0, 0, :4] = [0, 1, 2, 3]
    c[0, 1, 16, 130] = 2                     # W, row 16 (second row tile), code 130
    w = O.pack_codes(c)
    # 2 matrices x 2 row tiles x 2 chunks x 16 rows x 8 words
    assert w.shape == (2 * 2 * 2 * 128,)
    # Re+Im < 0 for codes 2, 3 -> bits 1 (even code 2) and 9 (odd code 3);
    # Re-Im < 0 for codes 1, 2 -> bits 16+8 (odd code 1) and 16+1 (even code 2)
    assert w[0] == 0x01020202
    # W (block 4), row tile 1, chunk 1 (codes 128..255), row 0, word 0, lane 2
    idx = (((1 * 2 + 1) * 2 + 1) * 16 + 0) * 8 + 0
    assert w[idx] == (1 << 1) | (1 << 17)
    assert np.count_nonzero(w) == 2


@pytest.mark.parametrize("T,n,m", [(1, 16, 128), (2, 32, 256), (3, 5, 77), (2, 17, 129)])
def test_storage_is_T_bits_per_real_parameter(T, n, m):
    c = rng.integers(0, 4, (T, 2, n, m)).astype(np.uint8)
    w = O.pack_codes(c)
    assert np.array_equal(O.unpack_codes(w, T, n, m), c)
    if m % 128 == 0 and n % 16 == 0:
        assert w.nbytes * 8 == T * (2 * n) * (2 * m)     # T bits per real parameter of R


# ---------------------------------------------------------------- quantized matmul
@pytest.mark.parametrize("rows,cols,T", [(8, 8, 1), (7, 9, 2), (32, 20, 3), (5, 130, 2)])
def test_wl_matmul_equals_dense_realified(rows, cols, T):
    """Two independent formulas: complex sum_t (U^t x + W^t conj x) vs dense real R^ x~."""
    R = 0.02 * rng.standard_normal((rows, cols)).astype(np.float32)
    U, W = O.convert(R)
    codes, scales = O.quantize(U, W, T)
    x = rng.standard_normal((3, cols))
    y = O.wl_matmul(x, codes, scales, rows)
    n, m = U.shape
    xp = np.zeros((3, 2 * m))
    xp[:, :cols] = x
    y2 = (O.dense_realified(codes, scales) @ xp.T).T[:, :rows]
    assert np.max(np.abs(y - y2)) <= 1e-12 * max(1.0, np.abs(y2).max())


def test_wl_matmul_all_plus_one():
    n, m = 6, 10
    codes = np.zeros((1, 2, n, m), dtype=np.uint8)
    scales = np.array([[[0.5, 7.0], [0.25, 9.0]]], dtype=np.float32)
    x = rng.standard_normal((2, 2 * m))
    z = x[:, :m] + 1j * x[:, m:]
    y = O.wl_matmul(x, codes, scales, 2 * n)
    expect = 0.5 * z.sum(axis=1) + 0.25 * np.conj(z).sum(axis=1)
    assert np.allclose(y[:, :n], expect.real[:, None], atol=1e-13)
    assert np.allclose(y[:, n:], expect.imag[:, None], atol=1e-13)


def test_wl_matmul_plus_i_uses_s_im():
    """Codes +i on W only: y = i s_im^W sum conj(x); s_re must not enter (Algorithm 1 read with
    Eq. ifairy-dequant's scale placement)."""
    n, m = 3, 5
    codes = np.zeros((1, 2, n, m), dtype=np.uint8)
    codes[0, 1] = 1
    scales = np.array([[[0.0, 0.0], [100.0, 3.0]]], dtype=np.float32)
    x = rng.standard_normal((1, 2 * m))
    z = x[:, :m] + 1j * x[:, m:]
    expect = 1j * 3.0 * np.conj(z).sum(axis=1)
    y = O.wl_matmul(x, codes, scales, 2 * n)
    assert np.allclose(y[:, :n], expect.real[:, None]) and np.allclose(y[:, n:], expect.imag[:, None])


def test_dequant_each_codeword_by_hand():
    """Eq. ifairy-dequant with hand-written codewords i^c: c = 0 -> +1, 1 -> +i, 2 -> -1,
    3 -> -i, the real part scaled by s_re and the imaginary part by s_im (s_re != s_im, so a
    swapped scale or a wrong sign on any codeword fails)."""
    s_re, s_im = np.float32(0.375), np.float32(2.5)
    got = O.dequant(np.array([0, 1, 2, 3]), s_re, s_im)
    want = np.array([0.375 + 0j, 2.5j, -0.375 + 0j, -2.5j])
    assert np.array_equal(got, want)


@pytest.mark.parametrize("shape", [(9, 14), (1, 1), (32, 5)])
def test_dequant_is_the_residual_step(shape):
    """R^(t) - dequant(B^(t), s^(t)) = R^(t+1) exactly (math mode): dequant agrees with the
    residual update of Sec. 3.3, whose scales are pinned by the norm identity above."""
    M = rng.standard_normal(shape) + 1j * rng.standard_normal(shape)
    codes, scales, res = O.residual_quantize(M, 3, mode="math")
    for t in range(3):
        r = res[t][0] + 1j * res[t][1]
        nxt = res[t + 1][0] + 1j * res[t + 1][1]
        assert np.array_equal(r - O.dequant(codes[t], scales[t][0], scales[t][1]), nxt)


@pytest.mark.parametrize("mat,code", [(0, 2), (0, 3), (1, 2), (1, 3)])
def test_wl_matmul_minus_codes_closed_form(mat, code):
    """All codes -1 (c = 2) or -i (c = 3) on one matrix, a large scale on the unused axis that
    must not appear: U with -1 gives y = -s_re sum x, U with -i gives y = -i s_im sum x; on W the
    same with conj(x) (Eq. widely-linear)."""
    n, m = 4, 7
    codes = np.zeros((1, 2, n, m), dtype=np.uint8)
    codes[0, mat] = code
    scales = np.zeros((1, 2, 2), dtype=np.float32)
    s_used, s_unused = 0.625, 1000.0
    scales[0, mat] = (s_used, s_unused) if code == 2 else (s_unused, s_used)
    x = rng.standard_normal((2, 2 * m))
    z = x[:, :m] + 1j * x[:, m:]
    zz = z if mat == 0 else np.conj(z)
    factor = -s_used if code == 2 else -1j * s_used
    expect = factor * zz.sum(axis=1)
    y = O.wl_matmul(x, codes, scales, 2 * n)
    assert np.allclose(y[:, :n], expect.real[:, None], atol=1e-12)
    assert np.allclose(y[:, n:], expect.imag[:, None], atol=1e-12)


def test_unquantized_limit_is_theorem1():
    """Replacing the dequantized matrices by U, W reproduces R x~."""
    R = rng.standard_normal((10, 14))
    U, W = O.convert(R, mode="math")
    x = rng.standard_normal((2, 14))
    z = O.split_input(x, U.shape[1])
    y = z @ U.T + np.conj(z) @ W.T
    assert np.allclose(np.concatenate([y.real, y.imag], 1), x @ R.T, atol=1e-12)


def test_tolerance_bound_bounds_y():
    R = 0.02 * rng.standard_normal((64, 64)).astype(np.float32)
    U, W = O.convert(R)
    codes, scales = O.quantize(U, W, 2)
    x = rng.standard_normal((4, 64))
    y = O.wl_matmul(x, codes, scales, 64)
    n = 32
    mag = np.abs(y[:, :n] + 1j * y[:, n:])
    assert np.all(mag.max(axis=1) <= O.tolerance_bound(x, scales) * (1 + 1e-12))


# ------------------------------------------------------------------ adjoint (input gradient)
@pytest.mark.parametrize("n,m,T", [(3, 5, 1), (4, 4, 2), (7, 2, 3), (1, 9, 2)])
def test_adjoint_codes_realify_to_the_transpose(n, m, T):
    """The adjoint codes realify (Eq. realify-ops, Eq. R-sum) to exactly the transpose of the
    original layer's real map, for every code value in U and in W (a missing conjugation, a
    conjugated W or an untransposed block fails)."""
    g = np.random.default_rng(n * 31 + m * 7 + T)
    codes = g.integers(0, 4, (T, 2, n, m)).astype(np.uint8)
    scales = (0.01 + 0.03 * g.random((T, 2, 2))).astype(np.float32)
    Rh = O.dense_realified(codes, scales)
    Ra = O.dense_realified(O.adjoint_codes(codes), scales)
    assert Ra.shape == (2 * m, 2 * n)
    assert np.array_equal(Ra, Rh.T)


def test_adjoint_codes_are_an_involution():
    g = np.random.default_rng(5)
    codes = g.integers(0, 4, (3, 2, 6, 11)).astype(np.uint8)
    assert np.array_equal(O.adjoint_codes(O.adjoint_codes(codes)), codes)


@pytest.mark.parametrize("out_f,in_f", [(6, 10), (7, 9), (9, 4)])
def test_adjoint_matmul_is_the_input_gradient(out_f, in_f):
    """<R^ x~, g~> = <x~, wl_matmul(g~, adjoint codes)> for the real layouts, odd sizes included
    (the padded output channel carries no gradient)."""
    g = np.random.default_rng(out_f + 10 * in_f)
    n, m = O.complex_dims(out_f, in_f)
    codes = g.integers(0, 4, (2, 2, n, m)).astype(np.uint8)
    scales = (0.01 + 0.03 * g.random((2, 2, 2))).astype(np.float32)
    x = g.standard_normal((3, in_f))
    gy = g.standard_normal((3, out_f))
    y = O.wl_matmul(x, codes, scales, out_f)
    gx = O.wl_matmul(gy, O.adjoint_codes(codes), scales, in_f)
    assert np.allclose(np.sum(y * gy, axis=1), np.sum(x * gx, axis=1), rtol=1e-12, atol=1e-12)
    Rh = O.dense_realified(codes, scales)[:out_f, :in_f]
    assert np.allclose(gx, gy @ Rh, rtol=1e-12, atol=1e-12)
