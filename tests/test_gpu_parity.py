"""GPU parity: the CUDA library (through its C ABI) against the CPU oracle on the same seeded
inputs. Conversion, codes and scales must match bit for bit; matmul outputs must satisfy
relative Frobenius error <= 1e-5 and |err| <= 1e-4 * ||x~||_1 * sum_t s_t per element, where
sum_t s_t = sum over stages of max(s_re, s_im) of U plus that of W."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2512_02901_gb300 import synth

pytestmark = pytest.mark.gpu

REL_FRO = 1e-5
ELEM = 1e-4


@pytest.fixture(scope="module")
def F():
    import __graft_entry__ as entry
    entry.build()
    from paper_2512_02901_gb300 import binding
    binding.load()
    return binding


DEV = "cuda:0"


def _np_codes(codes_t):
    return codes_t.cpu().numpy().view(np.uint32).reshape(-1)


def assert_wl_close(yg, yo, x, scales, rows=None):
    yg = np.asarray(yg, dtype=np.float64)
    err = yg - yo
    denom = np.linalg.norm(yo)
    rel = np.linalg.norm(err) / denom if denom > 0 else np.linalg.norm(err)
    assert rel <= REL_FRO, f"relative Frobenius error {rel:.3e}"
    bound = ELEM * O.tolerance_bound(np.asarray(x, np.float64), scales)[:, None]
    worst = np.max(np.abs(err) - bound)
    assert worst <= 0, f"element error exceeds bound by {worst:.3e}"


def upload_codes(packed):
    return torch.from_numpy(np.ascontiguousarray(packed).view(np.int32)).to(DEV)


# ------------------------------------------------------------------------------ convert
@pytest.mark.parametrize("rows,cols", [(256, 256), (7, 9), (1, 1), (3, 130), (4096, 4096),
                                       (11008, 4096), (4096, 11008)])
def test_convert_bit_exact(F, rows, cols):
    R = synth.random_matrix(rows, cols, seed=rows * 7 + cols, scale=0.02)
    U, W = F.convert(R.to(DEV))
    Uo, Wo = O.convert(R.numpy())
    assert np.array_equal(U.cpu().numpy().view(np.uint64), Uo.view(np.uint64))
    assert np.array_equal(W.cpu().numpy().view(np.uint64), Wo.view(np.uint64))


def test_convert_strided_input(F):
    base = synth.random_matrix(10, 40, seed=5)
    R = base[:, 3:20]                                    # ldR = 40 > cols = 17
    U, W = F.convert(base.to(DEV)[:, 3:20])
    Uo, Wo = O.convert(R.contiguous().numpy())
    assert np.array_equal(U.cpu().numpy(), Uo) and np.array_equal(W.cpu().numpy(), Wo)


# ------------------------------------------------------------------------------ quantize
def _quantize_both(F, U_np, W_np, T):
    U = torch.from_numpy(U_np).to(DEV)
    W = torch.from_numpy(W_np).to(DEV)
    codes, scales = F.quantize(U, W, T)
    assert F.get_status() == 0
    co, so = O.quantize(U_np, W_np, T)
    return codes, scales, co, so


def _assert_quant_equal(codes, scales, co, so):
    got = _np_codes(codes)
    want = O.pack_codes(co)
    assert got.shape == want.shape
    mism = np.argwhere(got != want)
    assert mism.size == 0, f"{len(mism)} packed words differ, first at {mism[:3].tolist()}"
    gs = scales.cpu().numpy()
    assert np.array_equal(gs.view(np.uint32), so.view(np.uint32)), (gs, so)


@pytest.mark.parametrize("n,m,T", [(128, 128, 2), (37, 53, 3), (1, 1, 1), (5, 65, 2), (300, 17, 4),
                                   (64, 200, 8)])
def test_quantize_bit_exact_small(F, n, m, T):
    g = np.random.default_rng(n * 1000 + m)
    U = (0.02 * g.standard_normal((n, m)) + 0.02j * g.standard_normal((n, m))).astype(np.complex64)
    W = (0.02 * g.standard_normal((n, m)) + 0.02j * g.standard_normal((n, m))).astype(np.complex64)
    _assert_quant_equal(*_quantize_both(F, U, W, T))


def test_quantize_tiny_layer_bit_exact(F):
    A, _ = synth.tiny_layer()
    U, W = F.convert(A.to(DEV))
    codes, scales = F.quantize(U, W, 2)
    Uo, Wo = O.convert(A.numpy())
    co, so = O.quantize(Uo, Wo, 2)
    _assert_quant_equal(codes, scales, co, so)


def test_quantize_ties_zero_and_degenerate(F):
    """Exact ties, signed zeros, an all-zero matrix (empty +-i set -> s_im = 0)."""
    vals = np.array([1, -1, 0.5, -0.5, 0.0, -0.0, 2.0], dtype=np.float32)
    g = np.random.default_rng(7)
    re = g.choice(vals, size=(19, 33)).astype(np.float32)
    im = np.where(g.random((19, 33)) < 0.5, re, -re).astype(np.float32)
    U = (re + 1j * im).astype(np.complex64)
    W = np.zeros((19, 33), dtype=np.complex64)
    codes, scales, co, so = _quantize_both(F, U, W, 3)
    _assert_quant_equal(codes, scales, co, so)
    assert so[0, 1, 1] == 0.0


def test_quantize_strided_rows(F):
    g = np.random.default_rng(11)
    big = (g.standard_normal((20, 80)) + 1j * g.standard_normal((20, 80))).astype(np.complex64)
    Ud = torch.from_numpy(big).to(DEV)[:, :70]
    Wd = torch.from_numpy(big[:, ::-1].copy()).to(DEV)[:, :70]
    codes, scales = F.quantize(Ud, Wd, 2)
    co, so = O.quantize(big[:, :70], big[:, ::-1][:, :70], 2)
    _assert_quant_equal(codes, scales, co, so)


def test_quantize_nonfinite_latches_status(F):
    U = torch.zeros((4, 16), dtype=torch.complex64, device=DEV)
    U[1, 3] = complex(float("nan"), 0.0)
    W = torch.ones((4, 16), dtype=torch.complex64, device=DEV)
    F.quantize(U, W, 1)
    assert F.get_status() == 6
    assert F.get_status() == 0          # read clears


def test_quantize_wide_range_values(F):
    """Values spread over ~60 binades (and some subnormal): most 256-element groups take the
    float64 tree instead of the exact integer sum, some groups mix both cases across the two
    sums; codes and scales still bit-exact."""
    g = np.random.default_rng(21)
    n, m = 96, 1000
    def wide():
        mag = g.standard_normal((n, m)) * np.exp2(g.integers(-40, 21, (n, m)))
        mag[g.random((n, m)) < 0.01] = 3e-42            # float32 subnormals
        return mag
    U = (wide() + 1j * 0.02 * g.standard_normal((n, m))).astype(np.complex64)
    W = (0.02 * g.standard_normal((n, m)) + 1j * wide()).astype(np.complex64)
    _assert_quant_equal(*_quantize_both(F, U, W, 3))


def test_quantize_three_reduction_levels(F):
    """n m > 2^24: more than 256 level-1 groups, so the scales take a third tree level."""
    g = np.random.default_rng(23)
    n, m = 4100, 4100
    U = (0.02 * g.standard_normal((n, m)) + 0.02j * g.standard_normal((n, m))).astype(np.complex64)
    W = (0.02 * g.standard_normal((n, m)) - 0.01j * g.standard_normal((n, m))).astype(np.complex64)
    _assert_quant_equal(*_quantize_both(F, U, W, 1))


@pytest.mark.parametrize("rows,cols,T,seed", [
    (4096, 4096, 2, synth.weight_seed("attn")),             # attention projection, decode
    (11008, 4096, 2, synth.weight_seed("mlp", 0)),          # up / gate
    (4096, 11008, 2, synth.weight_seed("mlp", 2)),          # down
    (11008, 4096, 3, synth.weight_seed("prefill", 0)),
    (4096, 11008, 1, synth.weight_seed("prefill", 1)),
])
def test_quantize_bit_exact_full_size(F, rows, cols, T, seed):
    R = synth.student_t_weight(rows, cols, seed)
    U, W = F.convert(R.to(DEV))
    codes, scales = F.quantize(U, W, T)
    assert F.get_status() == 0
    Uo, Wo = O.convert(R.numpy())
    co, so = O.quantize(Uo, Wo, T)
    _assert_quant_equal(codes, scales, co, so)


# ------------------------------------------------------------------------------ wl_matmul
def _random_quantized(n, m, T, seed):
    g = np.random.default_rng(seed)
    codes = g.integers(0, 4, (T, 2, n, m)).astype(np.uint8)
    scales = (0.01 + 0.02 * g.random((T, 2, 2))).astype(np.float32)
    return codes, scales


def _run_wl(F, x_t, codes, scales, out_features, path=0):
    y = F.wl_matmul(x_t.to(DEV), upload_codes(O.pack_codes(codes)),
                    torch.from_numpy(scales).to(DEV), out_features, path=path)
    assert F.get_status() == 0
    return y.cpu().numpy()


def test_wl_tiny_layer_fp32(F):
    A, x = synth.tiny_layer()
    Uo, Wo = O.convert(A.numpy())
    co, so = O.quantize(Uo, Wo, 2)
    yg = _run_wl(F, x, co, so, 256)
    yo = O.wl_matmul(x.numpy(), co, so, 256)
    assert_wl_close(yg, yo, x.numpy(), so)


@pytest.mark.parametrize("out_f,in_f,T,B,dtype", [
    (8, 8, 1, 1, torch.float32), (37, 53, 2, 3, torch.float32), (37, 53, 3, 5, torch.bfloat16),
    (130, 258, 2, 17, torch.bfloat16), (1, 1, 1, 2, torch.float32), (2, 129, 8, 4, torch.bfloat16),
    (255, 1001, 2, 1, torch.bfloat16), (1024, 96, 2, 64, torch.bfloat16),
])
def test_wl_matmul_shapes(F, out_f, in_f, T, B, dtype):
    n, m = O.complex_dims(out_f, in_f)
    codes, scales = _random_quantized(n, m, T, seed=out_f * 31 + in_f)
    x = synth.random_matrix(B, in_f, seed=B + in_f).to(dtype)
    yg = _run_wl(F, x, codes, scales, out_f)
    xo = x.float().numpy()
    yo = O.wl_matmul(xo, codes, scales, out_f)
    assert_wl_close(yg, yo, xo, scales)


def test_wl_matmul_strided_x_and_y(F):
    n, m, T, B = 40, 24, 2, 6
    codes, scales = _random_quantized(n, m, T, seed=3)
    xbig = synth.random_matrix(B, 2 * m + 16, seed=9).to(torch.bfloat16)
    x = xbig.to(DEV)[:, : 2 * m]
    y = torch.full((B, 2 * n + 8), 7.0, device=DEV)
    F.wl_matmul(x, upload_codes(O.pack_codes(codes)), torch.from_numpy(scales).to(DEV), 2 * n,
                y=y[:, : 2 * n])
    yg = y.cpu().numpy()
    assert np.all(yg[:, 2 * n:] == 7.0)                      # beyond out_features untouched
    xo = xbig[:, : 2 * m].float().numpy()
    assert_wl_close(yg[:, : 2 * n], O.wl_matmul(xo, codes, scales, 2 * n), xo, scales)


def _layer(rows, cols, T, seed):
    R = synth.student_t_weight(rows, cols, seed)
    Uo, Wo = O.convert(R.numpy())
    co, so = O.quantize(Uo, Wo, T)
    return co, so


@pytest.mark.parametrize("rows,cols,B,seed", [
    (4096, 4096, 1, synth.weight_seed("attn")),
    (11008, 4096, 1, synth.weight_seed("mlp", 0)),
    (11008, 4096, 4, synth.weight_seed("mlp", 1)),
    (4096, 11008, 16, synth.weight_seed("mlp", 2)),
])
def test_wl_matmul_full_size_decode(F, rows, cols, B, seed):
    co, so = _layer(rows, cols, 2, seed)
    x = synth.outlier_activations(B, cols, synth.activation_seed(seed, B))
    yg = _run_wl(F, x, co, so, rows)
    xo = x.float().numpy()
    yo = O.wl_matmul(xo, co, so, rows)
    assert_wl_close(yg, yo, xo, so)


@pytest.mark.parametrize("rows,cols,T", [(11008, 4096, 1), (11008, 4096, 2), (11008, 4096, 3),
                                         (4096, 11008, 1), (4096, 11008, 2), (4096, 11008, 3)])
def test_wl_matmul_prefill_sampled(F, rows, cols, T):
    """2048 tokens through the default path (the tcgen05 prefill GEMM), every (layer, T) pair the
    benchmark times; the oracle computes a sample of 96 output rows for every token."""
    seed = synth.weight_seed("prefill", 0 if rows > cols else 1)
    co, so = _layer(rows, cols, T, seed)
    B = 2048
    x = synth.outlier_activations(B, cols, synth.activation_seed(seed, B))
    yg = _run_wl(F, x, co, so, rows)
    n, m = co.shape[2], co.shape[3]
    g = np.random.default_rng(0)
    rws = np.sort(g.choice(n, 96, replace=False))
    xo = x.float().numpy()
    yc = O.wl_matmul_rows(O.split_input(xo, m), co, so, rws)
    yo = np.concatenate([yc.real, yc.imag], axis=1)
    ys = np.concatenate([yg[:, rws], yg[:, n + rws]], axis=1)
    assert_wl_close(ys, yo, xo, so)


@pytest.mark.parametrize("out_f,in_f,T,B", [
    (32, 32, 1, 1), (31, 515, 2, 2), (4096, 4096, 4, 1), (100, 8192, 3, 2), (17, 2, 2, 1),
    (4096, 11008, 2, 2), (11008, 4096, 2, 1), (48, 1024, 2, 2),
])
def test_wl_decode_path(F, out_f, in_f, T, B):
    """The decode path (tensor-core GEMV for B <= 2 bf16 tokens) on ragged rows and chunks."""
    n, m = O.complex_dims(out_f, in_f)
    codes, scales = _random_quantized(n, m, T, seed=out_f + 7 * in_f + T)
    x = synth.outlier_activations(B, in_f, seed=out_f + in_f)
    yg = _run_wl(F, x, codes, scales, out_f, path=1)
    xo = x.float().numpy()
    assert_wl_close(yg, O.wl_matmul(xo, codes, scales, out_f), xo, scales)


def test_wl_decode_all_codes_each_value(F):
    """Every code value in every word position (catches a wrong position class)."""
    n, m, T = 16, 256, 1
    codes = np.zeros((T, 2, n, m), dtype=np.uint8)
    for j in range(n):
        codes[0, 0, j] = (np.arange(m) + j) % 4
        codes[0, 1, j] = (np.arange(m) // 16 + 3 * j) % 4
    scales = np.array([[[0.03, 0.011], [0.017, 0.029]]], dtype=np.float32)
    x = synth.outlier_activations(1, 2 * m, seed=99)
    yg = _run_wl(F, x, codes, scales, 2 * n, path=1)
    xo = x.float().numpy()
    assert_wl_close(yg, O.wl_matmul(xo, codes, scales, 2 * n), xo, scales)


# ------------------------------------------------------------------------------ retired path 2
def test_retired_path_2_is_rejected(F):
    """Path 2 (an earlier tcgen05 decode kernel, slower than both decode kernels that replaced
    it) is retired: every call naming it returns FAIRY2I_ERR_INVALID_ARG and enqueues nothing."""
    n, m, T = 16, 64, 2
    codes, scales = _random_quantized(n, m, T, seed=13)
    cd = upload_codes(O.pack_codes(codes))
    sc = torch.from_numpy(scales).to(DEV)
    for x in (synth.outlier_activations(1, 2 * m, seed=1).to(DEV),
              synth.outlier_activations(3, 2 * m, seed=1).to(DEV),
              torch.zeros((1, 2 * m), dtype=torch.float32, device=DEV)):
        with pytest.raises(F.Fairy2iError) as e:
            F.wl_matmul(x, cd, sc, 2 * n, path=2)
        assert e.value.code == 1
    assert F.get_status() == 0


# ------------------------------------------------------------------------------ tcgen05 prefill
@pytest.mark.parametrize("out_f,in_f,T,B", [
    (64, 256, 1, 64), (64, 256, 2, 3), (37, 144, 2, 70), (64, 256, 3, 130), (64, 256, 4, 64),
    (50, 272, 4, 9), (2, 16, 1, 5), (4096, 4096, 2, 64), (256, 2048, 2, 130), (96, 1024, 3, 200),
    (1000, 4096, 2, 65), (130, 400, 1, 129),
    # 32-token tiles (B <= 32, two issuing threads per sign plane): full, ragged, the boundary
    (4096, 4096, 2, 16), (11008, 4096, 2, 32), (4096, 11008, 3, 31), (300, 1024, 4, 17),
    (64, 256, 1, 33), (2048, 2048, 2, 1),
    # K split over CTA pairs (few tiles): 21 + 22 chunks, 2 + 3, 1 + 1, several tiles per pair
    (4096, 11008, 2, 64), (100, 1280, 4, 40), (130, 400, 1, 129), (11008, 4096, 3, 20),
    (1000, 2048, 1, 20), (4096, 4096, 1, 64), (200, 3008, 2, 7),
    # T = 3 from 512 tokens on: a T = 2 launch, then a T = 1 launch adding into y
    (300, 1024, 3, 600), (130, 400, 3, 512),
])
def test_wl_tcgen05_prefill_path(F, out_f, in_f, T, B):
    """The tcgen05 prefill GEMM (path 3): ragged row blocks (R = 64, 32, 16, 16 rows of every
    stage-matrix for T = 1..4), ragged token tiles (32 tokens up to a batch of 32, else 64),
    ragged 64-code x stages and 128-code chunks, one CTA or many tiles per CTA, and the K split
    over CTA pairs that launches of few tiles take."""
    n, m = O.complex_dims(out_f, in_f)
    codes, scales = _random_quantized(n, m, T, seed=5 * out_f + 3 * in_f + T)
    x = synth.outlier_activations(B, in_f, seed=out_f + in_f + 2)
    yg = _run_wl(F, x, codes, scales, out_f, path=3)
    xo = x.float().numpy()
    assert_wl_close(yg, O.wl_matmul(xo, codes, scales, out_f), xo, scales)


@pytest.mark.parametrize("B", [70, 20])
@pytest.mark.parametrize("T", [1, 2, 3, 4])
def test_wl_tcgen05_prefill_all_codes_each_value(F, T, B):
    """Every code value at every word position of every stage-matrix lane block, 70 tokens (64-token
    tiles) and 20 (32-token tiles)."""
    n, m = 40, 384
    codes = np.zeros((T, 2, n, m), dtype=np.uint8)
    for t in range(T):
        for j in range(n):
            codes[t, 0, j] = (np.arange(m) + j + t) % 4
            codes[t, 1, j] = (np.arange(m) // 16 + 3 * j + t) % 4
    g = np.random.default_rng(10 + T)
    scales = (0.01 + 0.02 * g.random((T, 2, 2))).astype(np.float32)
    x = synth.outlier_activations(B, 2 * m, seed=17 + T)
    yg = _run_wl(F, x, codes, scales, 2 * n, path=3)
    xo = x.float().numpy()
    assert_wl_close(yg, O.wl_matmul(xo, codes, scales, 2 * n), xo, scales)


def test_wl_tcgen05_prefill_strided_odd_input(F):
    """Odd in_features (the last Im channel padded) read through a row stride that keeps rows
    16-byte aligned; y written into a wider buffer."""
    m, T, B = 72, 2, 77
    in_f, n = 2 * m - 1, 45
    codes, scales = _random_quantized(n, m, T, seed=21)
    xbig = synth.outlier_activations(B, 152, seed=22)
    x = xbig.to(DEV)[:, :in_f]
    y = torch.full((B, 2 * n + 8), 7.0, device=DEV)
    F.wl_matmul(x, upload_codes(O.pack_codes(codes)), torch.from_numpy(scales).to(DEV), 2 * n,
                y=y[:, : 2 * n], path=3)
    assert F.get_status() == 0
    yg = y.cpu().numpy()
    assert np.all(yg[:, 2 * n:] == 7.0)
    xo = xbig[:, :in_f].float().numpy()
    assert_wl_close(yg[:, : 2 * n], O.wl_matmul(xo, codes, scales, 2 * n), xo, scales)


def test_wl_auto_path_routes_batches_to_prefill(F):
    """Above four tokens the default path is the prefill GEMM where it applies: same bits."""
    n, m, T, B = 300, 512, 2, 33
    codes, scales = _random_quantized(n, m, T, seed=23)
    cd = upload_codes(O.pack_codes(codes))
    sc = torch.from_numpy(scales).to(DEV)
    x = synth.outlier_activations(B, 2 * m, seed=24).to(DEV)
    y0 = F.wl_matmul(x, cd, sc, 2 * n, path=0)
    y3 = F.wl_matmul(x, cd, sc, 2 * n, path=3)
    assert F.get_status() == 0
    assert torch.equal(y0, y3)


def test_wl_tcgen05_prefill_rejects_outside_its_domain(F):
    n, m, T = 16, 64, 2
    codes, scales = _random_quantized(n, m, T, seed=25)
    cd = upload_codes(O.pack_codes(codes))
    sc = torch.from_numpy(scales).to(DEV)
    xs = [torch.zeros((8, 2 * m), dtype=torch.float32, device=DEV),                    # fp32 x
          synth.outlier_activations(8, 2 * m - 1, seed=2).to(DEV)]                     # ldx = 127
    for x in xs:
        with pytest.raises(F.Fairy2iError) as e:
            F.wl_matmul(x, cd, sc, 2 * n, path=3)
        assert e.value.code == 1
    codes5, scales5 = _random_quantized(n, m, 5, seed=26)                              # T = 5
    with pytest.raises(F.Fairy2iError) as e:
        F.wl_matmul(synth.outlier_activations(8, 2 * m, seed=3).to(DEV),
                    upload_codes(O.pack_codes(codes5)), torch.from_numpy(scales5).to(DEV),
                    2 * n, path=3)
    assert e.value.code == 1


# ------------------------------------------------------------------------------ failure detection
def test_bounded_wait_latches_timeout_and_context_survives(F):
    """A bounded wait on a barrier that nothing completes gives up after its limit, latches
    FAIRY2I_ERR_TIMEOUT, is cleared by reading it, and the context keeps working."""
    assert F.get_status() == 0
    F.selftest_wait_timeout(2000)                     # 2 ms
    assert F.get_status() == 7                        # FAIRY2I_ERR_TIMEOUT
    assert F.get_status() == 0                        # read and cleared
    n, m, T, B = 24, 40, 2, 3
    codes, scales = _random_quantized(n, m, T, seed=31)
    x = synth.random_matrix(B, 2 * m, seed=32)
    yg = _run_wl(F, x, codes, scales, 2 * n)
    xo = x.numpy()
    assert_wl_close(yg, O.wl_matmul(xo, codes, scales, 2 * n), xo, scales)


# ------------------------------------------------------------------------------ grouped linears
@pytest.mark.parametrize("out_f,in_f,T,B,count", [
    (4096, 4096, 2, 5, 3),      # q/k/v shapes at 5 tokens: one K-split launch
    (11008, 4096, 2, 8, 2),     # gate/up at 8 tokens
    (300, 1024, 3, 3, 2),       # ragged rows, T = 3
    (64, 256, 1, 2, 4),         # one 128-code chunk (no K split), four members
    (256, 1024, 2, 16, 4),      # four members, 16 tiles: K split over CTA pairs
])
def test_group_prefill_path_any_batch(F, out_f, in_f, T, B, count):
    """Path 3 for a group: one prefill GEMM launch holding every member's tiles, at skinny batches
    too; every member matches the oracle."""
    n, m = O.complex_dims(out_f, in_f)
    layers = [_random_quantized(n, m, T, seed=61 + 5 * g + out_f) for g in range(count)]
    x = synth.outlier_activations(B, in_f, seed=67 + in_f)
    xd = x.to(DEV)
    ys = F.wl_matmul_group(xd, [upload_codes(O.pack_codes(c)) for c, _ in layers],
                           [torch.from_numpy(s).to(DEV) for _, s in layers], out_f, path=3)
    assert F.get_status() == 0
    xo = x.float().numpy()
    for (c, s), yg in zip(layers, ys):
        assert_wl_close(yg.cpu().numpy(), O.wl_matmul(xo, c, s, out_f), xo, s)


@pytest.mark.parametrize("out_f,in_f,T,B,count,dtype", [
    (256, 512, 2, 1, 3, torch.bfloat16),      # one grouped decode launch (q, k, v shape class)
    (130, 258, 3, 2, 2, torch.bfloat16),      # ragged rows, two tokens
    (4096, 4096, 2, 1, 3, torch.bfloat16),    # the 7B attention projections
    (11008, 4096, 2, 1, 2, torch.bfloat16),   # the 7B gate and up projections
    (64, 256, 2, 4, 2, torch.bfloat16),       # 2 <= B <= 4: the chained kernel, one launch
    (64, 256, 2, 5, 2, torch.bfloat16),       # B > 4: one prefill launch for the group
    (64, 254, 2, 6, 2, torch.float32),        # float32 x at 6 tokens: the chained kernel, 4 + 2
    (64, 256, 2, 12, 2, torch.bfloat16),      # one prefill launch for the group
    (4096, 4096, 2, 64, 3, torch.bfloat16),   # the 7B q/k/v at 64 tokens: 192 tiles, one launch
    (11008, 4096, 2, 64, 2, torch.bfloat16),  # gate / up at 64 tokens: K split, 4-5 tiles a pair
    (300, 512, 3, 130, 2, torch.bfloat16),    # ragged rows, three token tiles
    (256, 512, 3, 520, 2, torch.bfloat16),    # T = 3 in two launches (stages 0-1, then 2)
    (37, 53, 2, 1, 4, torch.float32),         # fp32 x: members on the general path
])
def test_wl_matmul_group_equals_separate_calls(F, out_f, in_f, T, B, count, dtype):
    """A group of linears on one input gives the separate calls' results (bit for bit on the
    warp-MMA decode kernel, within the accumulation tolerance on the automatic path), and every
    member matches the oracle."""
    n, m = O.complex_dims(out_f, in_f)
    layers = [_random_quantized(n, m, T, seed=41 + 7 * g + out_f) for g in range(count)]
    x = synth.outlier_activations(B, in_f, seed=43 + in_f).to(dtype)
    xd = x.to(DEV)
    cds = [upload_codes(O.pack_codes(c)) for c, _ in layers]
    scs = [torch.from_numpy(s).to(DEV) for _, s in layers]
    ys = F.wl_matmul_group(xd, cds, scs, out_f)
    singles = [F.wl_matmul(xd, c, s, out_f) for c, s in zip(cds, scs)]
    # on the warp-MMA decode kernel (path 1) the group launch and the single calls run the same
    # arithmetic: bit for bit
    ys1p = F.wl_matmul_group(xd, cds, scs, out_f, path=1)
    singles1 = [F.wl_matmul(xd, c, s, out_f, path=1) for c, s in zip(cds, scs)]
    assert F.get_status() == 0
    xo = x.float().numpy()
    if B <= 2 and dtype == torch.bfloat16:     # where the warp-MMA kernel applies
        for a1, b1 in zip(ys1p, singles1):
            assert torch.equal(a1, b1)
    for g, (yg, ys1) in enumerate(zip(ys, singles)):
        # the automatic path may pick another decode kernel for the group than for a member
        assert torch.allclose(yg, ys1, rtol=1e-5, atol=1e-5 * float(ys1.abs().max()))
        if out_f * in_f <= 4096 * 4096 and g == 0:
            codes, scales = layers[g]
            assert_wl_close(yg.cpu().numpy(), O.wl_matmul(xo, codes, scales, out_f), xo, scales)


# ------------------------------------------------------------------------------ adjoint (input gradient)
@pytest.mark.parametrize("n,m,T", [(5, 9, 1), (16, 128, 2), (130, 300, 3), (257, 129, 4), (1, 1, 1),
                                   (2048, 5504, 2)])
def test_codes_adjoint_bit_exact(F, n, m, T):
    """Transposed, U-conjugated codes in the packed layout of an m x n layer, bit for bit."""
    codes, _ = _random_quantized(n, m, T, seed=n * 13 + m + T)
    got = F.codes_adjoint(upload_codes(O.pack_codes(codes)), n, m, T)
    assert F.get_status() == 0
    want = O.pack_codes(O.adjoint_codes(codes))
    assert np.array_equal(_np_codes(got), want)


@pytest.mark.parametrize("out_f,in_f,T,B,dtype", [
    (4096, 4096, 2, 1, torch.bfloat16),      # decode kernel on the adjoint codes
    (129, 258, 3, 2, torch.bfloat16),
    (64, 512, 2, 70, torch.bfloat16),        # prefill kernel
    (37, 53, 2, 3, torch.float32),           # general kernel, odd sizes
])
def test_input_gradient_through_adjoint_codes(F, out_f, in_f, T, B, dtype):
    """x~_grad = R^T y~_grad through the adjoint codes and the ordinary matmul paths."""
    n, m = O.complex_dims(out_f, in_f)
    codes, scales = _random_quantized(n, m, T, seed=out_f + 3 * in_f)
    adj = F.codes_adjoint(upload_codes(O.pack_codes(codes)), n, m, T)
    gy = synth.outlier_activations(B, out_f, seed=out_f * 5 + B).to(dtype)
    gx = F.wl_matmul(gy.to(DEV), adj, torch.from_numpy(scales).to(DEV), in_f)
    assert F.get_status() == 0
    go = gy.float().numpy()
    want = O.wl_matmul(go, O.adjoint_codes(codes), scales, in_f)
    assert_wl_close(gx.cpu().numpy(), want, go, scales)


# ------------------------------------------------------------------------------ stream ordering
@pytest.mark.parametrize("path", [1, 4])
def test_quantize_then_decode_back_to_back(F, path):
    """The decode kernels read the codes and scales before their programmatic-launch wait. They
    rely on the quantize kernel that wrote them (launched just before on the same stream, no
    synchronization between) having ended first. Codes and scales start as garbage and each
    round rewrites them, so a decode that read them early would differ from the oracle."""
    out_f, in_f, T = 4096, 4096, 2
    R = synth.student_t_weight(out_f, in_f, seed=91)
    n, m = O.complex_dims(out_f, in_f)
    Uo, Wo = O.convert(R.numpy())
    co, so = O.quantize(Uo, Wo, T)
    xs = [synth.outlier_activations(1, in_f, seed=92 + i) for i in range(3)]
    Rd = R.to(DEV)
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        for x in xs:
            codes = torch.full((T, 2, (n + 15) // 16, F.words_per_row(m) // 8, 16, 8), -1,
                               dtype=torch.int32, device=DEV)
            scales = torch.full((T, 2, 2), float("nan"), device=DEV)
            U, W = F.convert(Rd, stream=stream)
            F.quantize(U, W, T, codes=codes, scales=scales, stream=stream)
            y = F.wl_matmul(x.to(DEV), codes, scales, out_f, path=path, stream=stream)
            stream.synchronize()
            xo = x.float().numpy()
            assert_wl_close(y.cpu().numpy(), O.wl_matmul(xo, co, so, out_f), xo, so)
    assert F.get_status(stream) == 0
