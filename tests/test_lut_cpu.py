"""The host look-up-table matmul (Sec. 3.4, LUT-based optimization for CPU) and its int8
activations, on the CPU (no GPU): the oracle's int8 quantizer pinned by its defining
properties, the library's quantizer bit for bit against it, and the table-lookup matmul against
the oracle's widely-linear matmul of the dequantized int8 token. The integer partial sums are
exact, so the only difference is the final float rounding: |err| <= 1e-6 ||delta xq||_1 sum_t s_t
per element and relative Frobenius <= 1e-6."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2512_02901_gb300 import binding as F

rng = np.random.default_rng(2024)


def test_int8_quantizer_pins():
    x = (rng.standard_normal(1001) * 3).astype(np.float32)
    q, d = O.quantize_activations_int8(x)
    assert d == np.float32(np.max(np.abs(x)) / np.float32(127))
    assert np.max(np.abs(q.astype(np.int32))) == 127
    assert np.all(np.abs(x.astype(np.float64) - q.astype(np.float64) * float(d)) <= 0.5 * float(d) * (1 + 1e-6))
    # round half to even: x / delta = 2.5 -> 2, 3.5 -> 4 (delta = 1)
    q2, d2 = O.quantize_activations_int8(np.array([127.0, 2.5, 3.5, -2.5], np.float32))
    assert d2 == 1.0 and list(q2) == [127, 2, 4, -2]
    q0, d0 = O.quantize_activations_int8(np.zeros(7, np.float32))
    assert d0 == 0 and not q0.any()


@pytest.mark.parametrize("n", [1, 9, 4096])
def test_library_quantizer_matches_oracle(n):
    x = torch.from_numpy((rng.standard_normal(n) * 5).astype(np.float32))
    xq, d = F.lut_quantize_x(x)
    qo, do = O.quantize_activations_int8(x.numpy())
    assert np.float32(d) == do
    assert np.array_equal(xq.numpy(), qo)


def _layer(out_f, in_f, T, seed):
    g = np.random.default_rng(seed)
    n, m = O.complex_dims(out_f, in_f)
    codes = g.integers(0, 4, (T, 2, n, m)).astype(np.uint8)
    scales = (0.01 + 0.02 * g.random((T, 2, 2))).astype(np.float32)
    return codes, scales


def _check(codes, scales, out_f, in_f, x, nthreads):
    T = codes.shape[0]
    xq, d = F.lut_quantize_x(torch.from_numpy(x))
    ct = torch.from_numpy(np.ascontiguousarray(O.pack_codes(codes)).view(np.int32))
    y = F.lut_matmul(xq, d, ct, torch.from_numpy(scales), out_f, T=T, nthreads=nthreads).numpy()
    xd = xq.numpy().astype(np.float64) * d
    want = O.wl_matmul(xd[None, :], codes, scales, out_f)[0]
    err = np.abs(y.astype(np.float64) - want)
    assert np.linalg.norm(err) <= 1e-6 * np.linalg.norm(want)
    bound = 1e-6 * O.tolerance_bound(xd[None, :], scales)[0]
    assert np.all(err <= bound)


@pytest.mark.parametrize("out_f,in_f,T,nthreads", [
    (32, 32, 1, 1), (31, 515, 2, 4), (64, 256, 3, 2), (17, 2, 2, 1), (130, 4100, 2, 8),
    (4096, 4096, 2, 16),
])
def test_lut_matmul_matches_oracle(out_f, in_f, T, nthreads):
    codes, scales = _layer(out_f, in_f, T, seed=out_f + in_f)
    x = (rng.standard_normal(in_f) * 2).astype(np.float32)
    _check(codes, scales, out_f, in_f, x, nthreads)


def test_lut_every_index_of_every_group():
    """Rows that walk through all 256 indices of each group position of a word (every code value
    at every code position), for U and W."""
    T, n, m = 1, 256, 128
    codes = np.zeros((T, 2, n, m), dtype=np.uint8)
    for j in range(n):
        for k in range(m):
            w, i = divmod(k, 16)
            g = (i % 2) * 2 + (i // 8)            # the group code i belongs to
            jj = (i % 8) // 2                      # its position inside the group
            codes[0, 0, j, k] = (j >> (2 * jj)) % 4 if g == w % 4 else (j + k) % 4
            codes[0, 1, j, k] = (3 * j + k // 16) % 4
    scales = np.array([[[0.3, 0.7], [0.11, 0.05]]], dtype=np.float32)
    x = (rng.standard_normal(2 * m) * 4).astype(np.float32)
    _check(codes, scales, 2 * n, 2 * m, x, 3)


def test_lut_validation():
    lib = F.load()
    assert lib.fairy2i_lut_workspace_bytes(0) == 0
    assert lib.fairy2i_lut_matmul(None, 1.0, 4, None, None, 4, 1, None, None, 0, 1) == 1
    x = torch.tensor([float("inf"), 1.0])
    with pytest.raises(F.Fairy2iError):
        F.lut_quantize_x(x)
