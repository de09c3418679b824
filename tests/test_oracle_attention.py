"""Pins of the oracle's Hermitian attention and decoder layer (no GPU): each checks the oracle
against something other than itself -- the real dot product of the stacked vectors (the identity
Sec. 3.1 states for Eq. hermitian-score), a hand-computed score, closed forms of softmax
attention, and a decoder layer written in real arithmetic from the dense realified matrices."""
import numpy as np
import pytest

import oracle as O

rng = np.random.default_rng(777)


def _stacked(z):
    return np.concatenate([z.real, z.imag])


def test_hermitian_score_hand_example():
    """q = (1+2i, 3-i), k = (2-i, i): Re(q^H k) = Re(-5i + (3i - 1)) = -1, d_k = 4 -> -1/2;
    the stacked vectors (1, 3, 2, -1).(2, 0, -1, 1) give the same -1."""
    q = np.array([1 + 2j, 3 - 1j])
    K = np.array([[2 - 1j, 1j]])
    assert O.hermitian_scores(q, K, 1)[0, 0] == -0.5


@pytest.mark.parametrize("n,heads,L", [(8, 1, 3), (64, 4, 9), (128, 8, 1)])
def test_hermitian_scores_equal_stacked_real_dot_products(n, heads, L):
    """Re(q_h^H k_h) = [Re q_h; Im q_h] . [Re k_h; Im k_h] per head (Sec. 3.1)."""
    q = rng.standard_normal(n) + 1j * rng.standard_normal(n)
    K = rng.standard_normal((L, n)) + 1j * rng.standard_normal((L, n))
    S = O.hermitian_scores(q, K, heads)
    dc = n // heads
    for h in range(heads):
        sl = slice(h * dc, (h + 1) * dc)
        for l in range(L):
            want = float(_stacked(q[sl]) @ _stacked(K[l, sl])) / np.sqrt(2 * dc)
            assert abs(S[h, l] - want) <= 1e-12 * max(1.0, abs(want))


def test_hermitian_scores_invariant_under_a_common_phase():
    q = rng.standard_normal(16) + 1j * rng.standard_normal(16)
    K = rng.standard_normal((5, 16)) + 1j * rng.standard_normal((5, 16))
    rot = np.exp(0.7j)
    assert np.allclose(O.hermitian_scores(rot * q, rot * K, 2), O.hermitian_scores(q, K, 2),
                       atol=1e-12)


def test_attention_single_key_returns_its_value():
    q = rng.standard_normal(32) + 1j * rng.standard_normal(32)
    K = rng.standard_normal((1, 32)) + 1j * rng.standard_normal((1, 32))
    V = rng.standard_normal((1, 32)) + 1j * rng.standard_normal((1, 32))
    assert np.allclose(O.hermitian_attention(q, K, V, 4), V[0], atol=1e-15)


def test_attention_equal_scores_average_the_values():
    q = np.zeros(16, dtype=np.complex128)            # every score 0
    K = rng.standard_normal((6, 16)) + 1j * rng.standard_normal((6, 16))
    V = rng.standard_normal((6, 16)) + 1j * rng.standard_normal((6, 16))
    assert np.allclose(O.hermitian_attention(q, K, V, 2), V.mean(axis=0), atol=1e-14)


@pytest.mark.parametrize("n,heads,L", [(32, 2, 7), (64, 8, 20)])
def test_attention_equals_real_attention_on_stacked_heads(n, heads, L):
    """The real and imaginary parts are aggregated with the same real weights: written with real
    stacked head vectors, real softmax and real value sums."""
    q = rng.standard_normal(n) + 1j * rng.standard_normal(n)
    K = rng.standard_normal((L, n)) + 1j * rng.standard_normal((L, n))
    V = rng.standard_normal((L, n)) + 1j * rng.standard_normal((L, n))
    got = O.hermitian_attention(q, K, V, heads)
    dc = n // heads
    for h in range(heads):
        sl = slice(h * dc, (h + 1) * dc)
        s = np.array([_stacked(q[sl]) @ _stacked(K[l, sl]) for l in range(L)]) / np.sqrt(2 * dc)
        p = np.exp(s - s.max())
        p = p / p.sum()
        o = sum(p[l] * _stacked(V[l, sl]) for l in range(L))
        assert np.allclose(_stacked(got[sl]), o, atol=1e-13)


def test_rmsnorm_and_silu_closed_forms():
    h = np.array([3.0, -4.0])                        # mean square 12.5
    w = np.array([1.0, 2.0])
    assert np.allclose(O.rmsnorm(h, w, 0.0), [3 / np.sqrt(12.5), -8 / np.sqrt(12.5)])
    x = rng.standard_normal(50)
    r = O.rmsnorm(x, np.ones(50), 0.0)
    assert abs(np.mean(r * r) - 1.0) < 1e-12
    assert O.silu_mul(np.array([0.0]), np.array([5.0]))[0] == 0.0
    assert np.isclose(O.silu_mul(np.array([2.0]), np.array([1.0]))[0], 2 / (1 + np.exp(-2.0)))


def _random_layer(d, dff, T, g):
    layer = {}
    for nm, out_f, in_f in (("q", d, d), ("k", d, d), ("v", d, d), ("o", d, d),
                            ("gate", dff, d), ("up", dff, d), ("down", d, dff)):
        n, m = O.complex_dims(out_f, in_f)
        layer[nm] = (g.integers(0, 4, (T, 2, n, m)).astype(np.uint8),
                     (0.01 + 0.02 * g.random((T, 2, 2))).astype(np.float32))
    layer["w_attn"] = 1.0 + 0.1 * g.standard_normal(d)
    layer["w_mlp"] = 1.0 + 0.1 * g.standard_normal(d)
    return layer


@pytest.mark.parametrize("L", [0, 5])
def test_decoder_layer_equals_real_arithmetic_layer(L):
    """The widely-linear decoder layer against the same layer in real arithmetic: every linear as
    the dense realified matrix R^ (Eq. realify-ops, Eq. R-sum), attention over real stacked head
    vectors (head h = channels h dc.. of the real and of the imaginary half), real softmax."""
    d, dff, heads, T, eps = 64, 96, 4, 2, 1e-5
    g = np.random.default_rng(L + 3)
    layer = _random_layer(d, dff, T, g)
    n = d // 2
    Kc = g.standard_normal((L, n)) + 1j * g.standard_normal((L, n))
    Vc = g.standard_normal((L, n)) + 1j * g.standard_normal((L, n))
    h = g.standard_normal(d)
    got, k_new, v_new = O.decoder_layer(h, layer, Kc, Vc, heads, eps)

    R = {nm: O.dense_realified(*layer[nm]) for nm in ("q", "k", "v", "o", "gate", "up", "down")}
    x = h / np.sqrt(np.mean(h * h) + eps) * layer["w_attn"]
    q, k, v = R["q"] @ x, R["k"] @ x, R["v"] @ x
    keys = np.vstack([np.hstack([Kc.real, Kc.imag]), k[None, :]])
    vals = np.vstack([np.hstack([Vc.real, Vc.imag]), v[None, :]])
    dc = n // heads
    a = np.zeros(d)
    for hh in range(heads):
        idx = np.r_[hh * dc:(hh + 1) * dc, n + hh * dc:n + (hh + 1) * dc]
        s = keys[:, idx] @ q[idx] / np.sqrt(2 * dc)
        p = np.exp(s - s.max())
        p /= p.sum()
        a[idx] = p @ vals[:, idx]
    h1 = h + R["o"] @ a
    x2 = h1 / np.sqrt(np.mean(h1 * h1) + eps) * layer["w_mlp"]
    gt, up = R["gate"] @ x2, R["up"] @ x2
    h2 = h1 + R["down"] @ (gt / (1 + np.exp(-gt)) * up)
    assert np.allclose(got, h2, rtol=1e-11, atol=1e-11)
    assert np.allclose(np.hstack([k_new.real, k_new.imag]), k, atol=1e-12)
    assert np.allclose(np.hstack([v_new.real, v_new.imag]), v, atol=1e-12)
