"""GPU parity of the skinny-batch decode (the chained kernel with 2 or 4 tokens per launch: the
automatic path for 2 <= B <= 4, and for 5 <= B <= 8 where the prefill GEMM does not apply, and
wl_matmul path 5 for any B) against the CPU oracle: every
token of ragged and full-size layers, T = 1..4, float32 and bf16 x, strided x and y, grouped
linears, launches of 4, 2 and 1 tokens, an x of extreme range in every token. Tolerance as
everywhere: relative Frobenius <= 1e-5 and |err| <= 1e-4 ||x~||_1 sum_t s_t per element."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2512_02901_gb300 import synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


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


def _tokens(B, in_f, seed, dtype):
    x = synth.outlier_activations(B, in_f, seed=seed)
    if dtype == torch.float32:
        x = x.float() * (1.0 + 1e-3 * torch.arange(in_f))
    # tokens of different magnitudes: each has its own fixed-point scale
    return (x.float() * torch.logspace(-3, 3, B)[:, None]).to(dtype)


@pytest.mark.parametrize("out_f,in_f,T,B,dtype,path", [
    (32, 32, 1, 2, torch.bfloat16, 0),
    (31, 515, 2, 3, torch.bfloat16, 0),       # ragged: launches of 2 + 1 tokens
    (64, 256, 3, 4, torch.float32, 0),
    (4096, 4096, 2, 4, torch.bfloat16, 0),    # the 7B attention projection, one launch of 4
    (4096, 4096, 4, 5, torch.bfloat16, 5),    # T = 4: 4 + 1
    (11008, 4096, 2, 8, torch.bfloat16, 5),   # gate / up: 4 + 4
    (4096, 11008, 2, 6, torch.bfloat16, 5),   # down (43 chunks per row): 4 + 2
    (100, 8192, 1, 7, torch.float32, 0),      # T = 1, long rows, float32 x (automatic): 4 + 2 + 1
    (64, 1000, 2, 6, torch.float32, 0),       # float32 x at 6 tokens (automatic): 4 + 2
    (130, 24576, 2, 4, torch.bfloat16, 5),    # the longest row the kernel takes
    (17, 2, 2, 2, torch.float32, 5),          # a single complex input
    (48, 1024, 3, 16, torch.bfloat16, 5),     # path 5 for any batch: four launches of 4
])
def test_skinny_matches_oracle(F, out_f, in_f, T, B, dtype, path):
    n, m = O.complex_dims(out_f, in_f)
    codes, scales = _random_quantized(n, m, T, seed=out_f * 7 + in_f + B)
    x = _tokens(B, in_f, seed=out_f + 3 * in_f + B, dtype=dtype)
    y = F.wl_matmul(x.to(DEV), _upload(codes), torch.from_numpy(scales).to(DEV), out_f,
                    path=path, T=T)
    assert F.get_status() == 0
    xo = x.float().numpy().astype(np.float64)
    _close(y.cpu().numpy(), O.wl_matmul(xo, codes, scales, out_f), xo, scales)


def test_skinny_strided_x_and_y(F):
    """Rows of x and y with leading dimensions larger than the features: only each token's first
    in_features entries are read and its first out_features entries written."""
    out_f, in_f, T, B = 300, 1000, 2, 4
    n, m = O.complex_dims(out_f, in_f)
    codes, scales = _random_quantized(n, m, T, seed=3)
    xb = torch.full((B, in_f + 24), float("nan"), dtype=torch.bfloat16)
    xb[:, :in_f] = _tokens(B, in_f, seed=5, dtype=torch.bfloat16)
    yb = torch.full((B, out_f + 9), -7.0, device=DEV)
    F.wl_matmul(xb.to(DEV)[:, :in_f], _upload(codes), torch.from_numpy(scales).to(DEV), out_f,
                y=yb[:, :out_f], T=T)
    assert F.get_status() == 0
    xo = xb[:, :in_f].float().numpy().astype(np.float64)
    _close(yb[:, :out_f].cpu().numpy(), O.wl_matmul(xo, codes, scales, out_f), xo, scales)
    assert torch.all(yb[:, out_f:] == -7.0)


@pytest.mark.parametrize("count,B,path", [(3, 4, 0), (2, 3, 0), (2, 8, 5), (2, 6, 5)])
def test_skinny_group_matches_oracle(F, count, B, path):
    out_f, in_f, T = 4096, 4096, 2
    n, m = O.complex_dims(out_f, in_f)
    layers = [_random_quantized(n, m, T, seed=40 + g) for g in range(count)]
    x = _tokens(B, in_f, seed=41, dtype=torch.bfloat16)
    ys = F.wl_matmul_group(x.to(DEV), [_upload(c) for c, _ in layers],
                           [torch.from_numpy(s).to(DEV) for _, s in layers], out_f, path=path)
    assert F.get_status() == 0
    xo = x.float().numpy().astype(np.float64)
    for (c, s), yg in zip(layers, ys):
        _close(yg.cpu().numpy(), O.wl_matmul(xo, c, s, out_f), xo, s)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_skinny_element_bound_for_extreme_x(F, dtype):
    """Each token as (1, tiny, tiny, ...) scaled by its own power of two, the tiny entries just
    under half a unit of the 2^-28 grid, every code +1: the rounding errors add up in every row
    and every output stays within the per-element bound."""
    T, out_f, in_f, B = 2, 4096, 11008, 4
    n, m = O.complex_dims(out_f, in_f)
    codes = np.zeros((T, 2, n, m), dtype=np.uint8)
    scales = np.full((T, 2, 2), 0.02, dtype=np.float32)
    x = torch.full((B, in_f), 0.99609375 * 2.0 ** -28, dtype=torch.float32)
    x[:, 0] = 1.0
    x *= torch.tensor([1.0, 2.0 ** -20, 2.0 ** 12, -1.0])[:, None]
    x = x.to(dtype)
    y = F.wl_matmul(x.to(DEV), _upload(codes), torch.from_numpy(scales).to(DEV), out_f)
    assert F.get_status() == 0
    xo = x.float().numpy().astype(np.float64)
    err = np.asarray(y.cpu().numpy(), np.float64) - O.wl_matmul(xo, codes, scales, out_f)
    bound = 1e-4 * O.tolerance_bound(xo, scales)[:, None]
    assert np.max(np.abs(err) - bound) <= 0, f"element error {np.max(np.abs(err) / bound):.3f} of the bound"


def test_skinny_tokens_are_independent(F):
    """A token's outputs do not depend on the other tokens of its launch: NaN-free tokens keep
    their results when a neighbour token is replaced (same launch shape)."""
    out_f, in_f, T, B = 4096, 4096, 2, 4
    n, m = O.complex_dims(out_f, in_f)
    codes, scales = _random_quantized(n, m, T, seed=9)
    cd, sc = _upload(codes), torch.from_numpy(scales).to(DEV)
    x = _tokens(B, in_f, seed=11, dtype=torch.bfloat16).to(DEV)
    y1 = F.wl_matmul(x, cd, sc, out_f)
    x2 = x.clone()
    x2[2] = -3.0 * x2[2]
    y2 = F.wl_matmul(x2, cd, sc, out_f)
    assert F.get_status() == 0
    for b in (0, 1, 3):
        assert torch.equal(y1[b], y2[b])
