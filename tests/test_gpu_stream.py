"""GPU parity of the persistent tcgen05 decode kernel (wl_matmul path 4, and the grouped call on
path 4) against the CPU oracle: ragged rows and chunks, every T it takes, one and two tokens,
x staged by bulk copy and by plain loads, K split over clusters of 1..8 CTAs, several row blocks
per cluster, strided x and y, grouped linears. Tolerance as everywhere: relative Frobenius
<= 1e-5 and |err| <= 1e-4 ||x~||_1 sum_t s_t per element."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2512_02901_gb300 import synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
PATH = 4


@pytest.fixture(scope="module")
def F():
    import __graft_entry__ as entry
    entry.build()
    from paper_2512_02901_gb300 import binding
    binding.load()
    return binding


def _close(yg, yo, x, scales):
    yg = np.asarray(yg, dtype=np.float64)
    err = yg - yo
    rel = np.linalg.norm(err) / np.linalg.norm(yo)
    assert rel <= 1e-5, f"relative Frobenius error {rel:.3e}"
    bound = 1e-4 * O.tolerance_bound(np.asarray(x, np.float64), scales)[:, None]
    worst = np.max(np.abs(err) - bound)
    assert worst <= 0, f"element error exceeds bound by {worst:.3e}"


def _upload(codes):
    return torch.from_numpy(np.ascontiguousarray(O.pack_codes(codes)).view(np.int32)).to(DEV)


def _random_quantized(n, m, T, seed):
    g = np.random.default_rng(seed)
    codes = g.integers(0, 4, (T, 2, n, m)).astype(np.uint8)
    scales = (0.01 + 0.02 * g.random((T, 2, 2))).astype(np.float32)
    return codes, scales


@pytest.mark.parametrize("out_f,in_f,T,B", [
    (32, 32, 1, 1),          # one chunk, one row block
    (31, 515, 2, 2),         # odd sizes: x by plain loads, ragged last chunk and row block
    (64, 256, 3, 1),         # T = 3: 96 of the 128 lanes
    (4096, 4096, 4, 1),      # T = 4
    (100, 8192, 3, 2),       # long rows, few row blocks: K split over clusters
    (17, 2, 2, 1),           # a single complex input
    (4096, 11008, 2, 2),     # the 7B down projection shape, two tokens
    (11008, 4096, 2, 1),     # 172 row blocks: several jobs per cluster
    (48, 1024, 2, 2),
    (4096, 4096, 2, 1),      # the 7B attention projection shape
    (130, 24576, 2, 1),      # the longest row the kernel takes (96 chunks, 12 per CTA)
    (8192, 2048, 1, 2),      # T = 1: 64-row blocks
])
def test_stream_decode_matches_oracle(F, out_f, in_f, T, B):
    n, m = O.complex_dims(out_f, in_f)
    codes, scales = _random_quantized(n, m, T, seed=5 * out_f + 3 * in_f + T)
    x = synth.outlier_activations(B, in_f, seed=out_f + in_f + 2)
    y = F.wl_matmul(x.to(DEV), _upload(codes), torch.from_numpy(scales).to(DEV), out_f, path=PATH)
    assert F.get_status() == 0
    xo = x.float().numpy()
    _close(y.cpu().numpy(), O.wl_matmul(xo, codes, scales, out_f), xo, scales)


@pytest.mark.parametrize("T", [1, 2, 3, 4])
def test_stream_all_codes_each_value(F, T):
    """Every code value at every word position of every stage-matrix lane block."""
    n, m = 40, 384
    codes = np.zeros((T, 2, n, m), dtype=np.uint8)
    for t in range(T):
        for j in range(n):
            codes[t, 0, j] = (np.arange(m) + j + t) % 4
            codes[t, 1, j] = (np.arange(m) // 16 + 3 * j + t) % 4
    g = np.random.default_rng(T)
    scales = (0.01 + 0.02 * g.random((T, 2, 2))).astype(np.float32)
    x = synth.outlier_activations(2, 2 * m, seed=17 + T)
    y = F.wl_matmul(x.to(DEV), _upload(codes), torch.from_numpy(scales).to(DEV), 2 * n, path=PATH)
    assert F.get_status() == 0
    xo = x.float().numpy()
    _close(y.cpu().numpy(), O.wl_matmul(xo, codes, scales, 2 * n), xo, scales)


def test_stream_strided_x_and_y(F):
    n, m, T, B = 70, 136, 2, 2
    codes, scales = _random_quantized(n, m, T, seed=21)
    xbig = synth.outlier_activations(B, 2 * m + 24, seed=22)
    x = xbig.to(DEV)[:, : 2 * m]
    y = torch.full((B, 2 * n + 8), 7.0, device=DEV)
    F.wl_matmul(x, _upload(codes), torch.from_numpy(scales).to(DEV), 2 * n, y=y[:, : 2 * n],
                path=PATH)
    assert F.get_status() == 0
    yg = y.cpu().numpy()
    assert np.all(yg[:, 2 * n:] == 7.0)                       # beyond out_features untouched
    xo = xbig[:, : 2 * m].float().numpy()
    _close(yg[:, : 2 * n], O.wl_matmul(xo, codes, scales, 2 * n), xo, scales)


def test_stream_repeated_calls_are_deterministic(F):
    """Back-to-back launches on one stream (the programmatic-launch overlap) give identical
    results: the cross-CTA sums run in a fixed rank order."""
    out_f, in_f, T = 4096, 4096, 2
    n, m = O.complex_dims(out_f, in_f)
    codes, scales = _random_quantized(n, m, T, seed=23)
    cd, sc = _upload(codes), torch.from_numpy(scales).to(DEV)
    xs = [synth.outlier_activations(1, in_f, seed=30 + i).to(DEV) for i in range(4)]
    ys = [F.wl_matmul(x, cd, sc, out_f, path=PATH) for x in xs * 3]
    assert F.get_status() == 0
    for i in range(4):
        assert torch.equal(ys[i], ys[i + 4]) and torch.equal(ys[i], ys[i + 8])
    xo = xs[1].cpu().float().numpy()
    _close(ys[1].cpu().numpy(), O.wl_matmul(xo, codes, scales, out_f), xo, scales)


@pytest.mark.parametrize("out_f,in_f,T,B,count", [
    (4096, 4096, 2, 1, 3),     # q, k, v of the 7B model in one launch
    (11008, 4096, 2, 1, 2),    # gate and up
    (130, 258, 3, 2, 2),       # ragged, two tokens
    (256, 512, 1, 1, 4),
])
def test_stream_group_matches_oracle(F, out_f, in_f, T, B, count):
    n, m = O.complex_dims(out_f, in_f)
    layers = [_random_quantized(n, m, T, seed=61 + 5 * g + out_f) for g in range(count)]
    x = synth.outlier_activations(B, in_f, seed=63 + in_f)
    xd = x.to(DEV)
    ys = F.wl_matmul_group(xd, [_upload(c) for c, _ in layers],
                           [torch.from_numpy(s).to(DEV) for _, s in layers], out_f, path=PATH)
    assert F.get_status() == 0
    xo = x.float().numpy()
    for g in range(count):
        codes, scales = layers[g]
        if out_f * in_f > 4096 * 4096 and g > 0:
            continue      # the oracle's time: the first member of the large shapes
        _close(ys[g].cpu().numpy(), O.wl_matmul(xo, codes, scales, out_f), xo, scales)


def test_stream_rejects_outside_its_domain(F):
    n, m, T = 16, 64, 2
    codes, scales = _random_quantized(n, m, T, seed=71)
    cd, sc = _upload(codes), torch.from_numpy(scales).to(DEV)
    for x in (synth.outlier_activations(3, 2 * m, seed=1).to(DEV),          # B = 3
              torch.zeros((1, 2 * m), dtype=torch.float32, device=DEV)):    # fp32 x
        with pytest.raises(F.Fairy2iError) as e:
            F.wl_matmul(x, cd, sc, 2 * n, path=PATH)
        assert e.value.code == 1
    # rows longer than the kernel's 96 chunks
    m2 = 12288 + 128
    codes2, scales2 = _random_quantized(2, m2, 1, seed=72)
    with pytest.raises(F.Fairy2iError) as e:
        F.wl_matmul(torch.zeros((1, 2 * m2), dtype=torch.bfloat16, device=DEV), _upload(codes2),
                    torch.from_numpy(scales2).to(DEV), 4, path=PATH)
    assert e.value.code == 1
    with pytest.raises(F.Fairy2iError) as e:    # a group path that does not exist
        F.wl_matmul_group(torch.zeros((1, 2 * m), dtype=torch.bfloat16, device=DEV), [cd], [sc],
                          2 * n, path=2)
    assert e.value.code == 1
    assert F.get_status() == 0


def test_automatic_decode_kernels(F):
    """The automatic path runs one token (bf16 x) on the persistent kernel's one-token form, 2 to
    4 tokens on the chained kernel (path 5) and 5 or more bf16 tokens on the prefill GEMM (path
    3), one launch for a whole group: bit for bit the results of the explicit paths (every
    kernel is deterministic for a given launch shape)."""
    out_f, in_f, T = 4096, 4096, 2
    n, m = O.complex_dims(out_f, in_f)
    layers = [_random_quantized(n, m, T, seed=81 + g) for g in range(3)]
    cds = [_upload(c) for c, _ in layers]
    scs = [torch.from_numpy(s).to(DEV) for _, s in layers]
    for B, path in ((1, PATH), (2, 5), (4, 5), (5, 3), (8, 3)):
        x = synth.outlier_activations(B, in_f, seed=83 + B).to(DEV)
        auto_group = F.wl_matmul_group(x, cds, scs, out_f)
        explicit = F.wl_matmul_group(x, cds, scs, out_f, path=path)
        for a, p in zip(auto_group, explicit):
            assert torch.equal(a, p)
        assert torch.equal(F.wl_matmul(x, cds[0], scs[0], out_f),
                           F.wl_matmul(x, cds[0], scs[0], out_f, path=path))
    assert F.get_status() == 0


@pytest.mark.parametrize("out_f,in_f,B,dtype", [
    (4096, 11008, 1, torch.bfloat16),    # the 7B down projection
    (11008, 4096, 1, torch.bfloat16),    # the 7B gate / up projections
    (4096, 4096, 2, torch.bfloat16),     # two tokens
    (4096, 11008, 1, torch.float32),     # float32 x: the chained kernel
    (4096, 4096, 2, torch.float32),
])
def test_automatic_decode_element_bound_for_extreme_x(F, out_f, in_f, B, dtype):
    """Every output of the automatic decode path stays within the per-element bound
    1e-4 |x~|_1 sum_t s_t whatever x is. Worst case for the fixed-point forms: x = (1, tiny,
    tiny, ...) with the tiny entries just under half a unit of the grid (2^-26 of the slice
    maximum for bf16 x, 2^-28 for float32 x; the second token scaled by 2^-10 with its own tiny
    entries), every code +1 so that the rounding errors add up in every row."""
    T = 2
    n, m = O.complex_dims(out_f, in_f)
    codes = np.zeros((T, 2, n, m), dtype=np.uint8)
    scales = np.full((T, 2, 2), 0.02, dtype=np.float32)
    unit = 2.0 ** -26 if dtype == torch.bfloat16 else 2.0 ** -28
    x = torch.full((B, in_f), 0.99609375 * unit, dtype=torch.float32)
    x[0, 0] = 1.0
    if B > 1:
        x[1] = 2.0 ** -10 * 0.99609375 * unit * 4
        x[1, 7] = -(2.0 ** -10)
    x = x.to(dtype)
    y = F.wl_matmul(x.to(DEV), _upload(codes), torch.from_numpy(scales).to(DEV), out_f)
    assert F.get_status() == 0
    xo = x.float().numpy().astype(np.float64)
    err = np.asarray(y.cpu().numpy(), np.float64) - O.wl_matmul(xo, codes, scales, out_f)
    bound = 1e-4 * O.tolerance_bound(xo, scales)[:, None]
    assert np.max(np.abs(err) - bound) <= 0, f"element error {np.max(np.abs(err) / bound):.3f} of the bound"


@pytest.mark.parametrize("tiny", [0.99609375 * 2.0**-24, 0.99609375 * 2.0**-26])
def test_stream_one_token_element_bound_for_extreme_x(F, tiny):
    """The one-token form holds each x entry to half a unit in 2^-26 of the largest |x| of the
    CTA's K slice, so the l1 error of x stays below 3072 2^-26 |x|_1 (a slice holds at most 3072
    real values) and the error of every output below the per-element bound 1e-4 |x~|_1 sum_t s_t,
    whatever x is. Worst case here: 152 row blocks of 1536-input rows (one CTA takes a whole row),
    x = (1, tiny, tiny, ...) with the tiny entries just under half a unit (2^-24 would fall off
    with twelve digits), every code +1 so that the errors add up in every row. The relative
    Frobenius criterion is not checked: no fixed precision meets it for every input."""
    T, out_f, in_f = 2, 9728, 3072
    n, m = O.complex_dims(out_f, in_f)
    codes = np.zeros((T, 2, n, m), dtype=np.uint8)
    scales = np.full((T, 2, 2), 0.02, dtype=np.float32)
    x = torch.full((1, in_f), tiny, dtype=torch.float32).to(torch.bfloat16)
    x[0, 0] = 1.0
    y = F.wl_matmul(x.to(DEV), _upload(codes), torch.from_numpy(scales).to(DEV), out_f, path=PATH)
    assert F.get_status() == 0
    xo = x.float().numpy().astype(np.float64)
    err = np.asarray(y.cpu().numpy(), np.float64) - O.wl_matmul(xo, codes, scales, out_f)
    bound = 1e-4 * O.tolerance_bound(xo, scales)[:, None]
    assert np.max(np.abs(err) - bound) <= 0, f"element error {np.max(np.abs(err) / bound):.3f} of the bound"
