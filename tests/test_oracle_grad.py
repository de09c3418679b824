"""Pins of the oracle's QAT gradients (no GPU), each against something other than the formula
it checks: the dense real gradient G = g~^T x~ mapped through R = R_lin(U) + R_conj(W) (Eq.
realify-ops), and central finite differences of the loss with the codes held fixed."""
import numpy as np
import pytest

import oracle as O

rng = np.random.default_rng(31337)


@pytest.mark.parametrize("out_f,in_f,B", [(6, 10, 3), (7, 9, 2), (8, 8, 1)])
def test_ste_weight_grad_equals_realified_gradient(out_f, in_f, B):
    """dL/dR = g~^T x~ for y~ = R x~; with R11 = Re U + Re W, R12 = Im W - Im U,
    R21 = Im U + Im W, R22 = Re U - Re W the chain rule gives dRe U = G11 + G22,
    dIm U = G21 - G12, dRe W = G11 - G22, dIm W = G12 + G21."""
    n, m = O.complex_dims(out_f, in_f)
    x = rng.standard_normal((B, in_f))
    g = rng.standard_normal((B, out_f))
    xp = np.zeros((B, 2 * m)); xp[:, :in_f] = x
    gp = np.zeros((B, 2 * n)); gp[:, :out_f] = g
    G = gp.T @ xp
    G11, G12, G21, G22 = G[:n, :m], G[:n, m:], G[n:, :m], G[n:, m:]
    dU, dW = O.ste_weight_grad(x, g, n, m)
    assert np.allclose(dU.real, G11 + G22) and np.allclose(dU.imag, G21 - G12)
    assert np.allclose(dW.real, G11 - G22) and np.allclose(dW.imag, G12 + G21)


def test_ste_weight_grad_finite_differences():
    """L = <g~, (R_lin(U) + R_conj(W)) x~> is linear in U, W: central differences are exact."""
    n, m, B = 3, 4, 2
    x = rng.standard_normal((B, 2 * m))
    g = rng.standard_normal((B, 2 * n))
    U = rng.standard_normal((n, m)) + 1j * rng.standard_normal((n, m))
    W = rng.standard_normal((n, m)) + 1j * rng.standard_normal((n, m))

    def loss(U, W):
        R = O.realify_lin(U) + O.realify_conj(W)
        return float(np.sum(g * (x @ R.T)))
    dU, dW = O.ste_weight_grad(x, g, n, m)
    eps = 1e-3
    for j in range(n):
        for k in range(m):
            for part, unit in ((0, 1.0), (1, 1j)):
                E = np.zeros((n, m), complex); E[j, k] = unit * eps
                fdU = (loss(U + E, W) - loss(U - E, W)) / (2 * eps)
                fdW = (loss(U, W + E) - loss(U, W - E)) / (2 * eps)
                assert abs(fdU - (dU[j, k].real if part == 0 else dU[j, k].imag)) < 1e-9
                assert abs(fdW - (dW[j, k].real if part == 0 else dW[j, k].imag)) < 1e-9


@pytest.mark.parametrize("T,shape", [(1, (4, 5)), (2, (6, 7)), (3, (5, 9))])
def test_scale_path_grad_finite_differences(T, shape):
    """Codes frozen at M0; L(M) = <dM, M^(M)> with M^ = sum_t dequant(codes_t, scales_t(M)) and
    the scales recomputed from M through the residual recursion (Eq. ifairy-scale, Sec. 3.3):
    the analytic gradient against central differences (L is smooth away from the kinks of |.|)."""
    M0 = rng.standard_normal(shape) + 1j * rng.standard_normal(shape)
    codes, scales0, _ = O.residual_quantize(M0, T, mode="math")
    dM = rng.standard_normal(shape) + 1j * rng.standard_normal(shape)

    def scales_of(M):
        r = M.copy()
        out = []
        for t in range(T):
            c = codes[t]
            on_re = (c == 0) | (c == 2)
            s_re = np.abs(r.real)[on_re].mean() if on_re.any() else 0.0
            s_im = np.abs(r.imag)[~on_re].mean() if (~on_re).any() else 0.0
            out.append((s_re, s_im))
            r = r - O.dequant(c, s_re, s_im)
        return out

    def loss(M):
        sc = scales_of(M)
        Mh = sum(O.dequant(codes[t], *sc[t]) for t in range(T))
        return float(np.sum(dM.real * Mh.real + dM.imag * Mh.imag))
    rhat, shat = O.scale_path_grad(M0, codes, scales0, dM)
    eps = 1e-6
    for j in range(shape[0]):
        for k in range(shape[1]):
            for unit, part in ((1.0, "re"), (1j, "im")):
                E = np.zeros(shape, complex); E[j, k] = unit * eps
                fd = (loss(M0 + E) - loss(M0 - E)) / (2 * eps)
                an = rhat[j, k].real if part == "re" else rhat[j, k].imag
                assert abs(fd - an) <= 1e-6 * max(1.0, abs(an)), (j, k, part, fd, an)
    # the total scale gradients: L is linear in the stage-(T-1) scales (no later stage)
    t = T - 1
    c = codes[t]
    b_re = np.select([c == 0, c == 2], [1.0, -1.0], 0.0)
    assert np.isclose(shat[t][0], np.sum(dM.real * b_re))
