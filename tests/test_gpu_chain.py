"""GPU parity of the chained decode kernel (fairy2i_wl_matmul_chain, and wl_matmul path 5 for one
call) against the CPU oracle: ragged rows and chunks, T = 1..4, float32 and bf16 tokens, grouped
linears, K split over clusters of 1..8 CTAs, chains of many calls whose inputs are the previous
call's outputs, extreme inputs. Tolerance as everywhere: relative Frobenius <= 1e-5 and
|err| <= 1e-4 ||x~||_1 sum_t s_t per element."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2512_02901_gb300 import synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
PATH = 5


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


def _token(in_f, seed, dtype):
    x = synth.outlier_activations(1, in_f, seed=seed)
    return x if dtype == torch.bfloat16 else x.float() * (1.0 + 1e-3 * torch.arange(in_f))


@pytest.mark.parametrize("out_f,in_f,T,dtype", [
    (32, 32, 1, torch.bfloat16),        # one chunk, one row block
    (31, 515, 2, torch.bfloat16),       # odd sizes: x by single loads, ragged chunk and row block
    (64, 256, 3, torch.float32),        # T = 3: half tiles, 48 of 64 lanes per plane
    (4096, 4096, 4, torch.bfloat16),    # T = 4
    (100, 8192, 3, torch.bfloat16),     # long rows, few row blocks
    (17, 2, 2, torch.float32),          # a single complex input
    (4096, 11008, 2, torch.bfloat16),   # the 7B down projection shape
    (11008, 4096, 2, torch.bfloat16),   # the 7B gate/up shape: several jobs per cluster
    (48, 1024, 2, torch.float32),
    (4096, 4096, 2, torch.bfloat16),    # the 7B attention projection shape
    (130, 24576, 1, torch.bfloat16),    # the longest row the kernel takes (K split >= 4)
    (8192, 2048, 1, torch.float32),     # T = 1: 32-row blocks, two tiles per stage-matrix
    (66, 300, 4, torch.float32),        # T = 4 with a ragged last half tile
])
def test_chain_single_call_matches_oracle(F, out_f, in_f, T, dtype):
    n, m = O.complex_dims(out_f, in_f)
    codes, scales = _random_quantized(n, m, T, seed=7 * out_f + 3 * in_f + T)
    x = _token(in_f, out_f + in_f + 5, dtype)
    y = F.wl_matmul(x.to(DEV), _upload(codes), torch.from_numpy(scales).to(DEV), out_f,
                    path=PATH)
    assert F.get_status() == 0
    xo = x.float().numpy()
    _close(y.cpu().numpy(), O.wl_matmul(xo, codes, scales, out_f), xo, scales)


@pytest.mark.parametrize("T", [1, 2, 3, 4])
def test_chain_all_codes_each_value(F, T):
    """Every code value at every word position of every stage-matrix lane block."""
    n, m = 40, 384
    codes = np.zeros((T, 2, n, m), dtype=np.uint8)
    for t in range(T):
        for j in range(n):
            codes[t, 0, j] = (np.arange(m) + j + t) % 4
            codes[t, 1, j] = (np.arange(m) // 16 + 3 * j + t) % 4
    g = np.random.default_rng(T)
    scales = (0.01 + 0.02 * g.random((T, 2, 2))).astype(np.float32)
    x = synth.outlier_activations(1, 2 * m, seed=7 + T)
    y = F.wl_matmul(x.to(DEV), _upload(codes), torch.from_numpy(scales).to(DEV), 2 * n,
                    path=PATH)
    assert F.get_status() == 0
    xo = x.float().numpy()
    _close(y.cpu().numpy(), O.wl_matmul(xo, codes, scales, 2 * n), xo, scales)


@pytest.mark.parametrize("out_f,in_f,T,count", [(4096, 4096, 2, 3), (11008, 4096, 2, 2),
                                                (70, 600, 3, 4), (33, 130, 1, 2)])
def test_chain_group_matches_oracle(F, out_f, in_f, T, count):
    n, m = O.complex_dims(out_f, in_f)
    layers = [_random_quantized(n, m, T, seed=out_f + in_f + 11 * g) for g in range(count)]
    x = synth.outlier_activations(1, in_f, seed=in_f + count)
    ys = F.wl_matmul_group(x.to(DEV), [_upload(c) for c, _ in layers],
                           [torch.from_numpy(s).to(DEV) for _, s in layers], out_f, path=PATH)
    assert F.get_status() == 0
    xo = x.float().numpy()
    for (codes, scales), y in zip(layers, ys):
        _close(y.cpu().numpy(), O.wl_matmul(xo, codes, scales, out_f), xo, scales)


def _chain_layers(shapes, T, seed):
    """(codes, scales, device codes, device scales) per linear of every call."""
    out = []
    for i, (count, out_f, in_f) in enumerate(shapes):
        n, m = O.complex_dims(out_f, in_f)
        call = []
        for g in range(count):
            codes, scales = _random_quantized(n, m, T, seed=seed + 97 * i + g)
            call.append((codes, scales, _upload(codes), torch.from_numpy(scales).to(DEV)))
        out.append(call)
    return out


# (linears, out_features, in_features) per call: two decoder-like layers at half size (every
# row at least 8 chunks, so that every cluster size applies)
SMALL_STACK = [(3, 2048, 2048), (1, 2048, 2048), (2, 5504, 2048), (1, 2048, 5504)] * 2


@pytest.mark.parametrize("cluster", [0, 1, 2, 4, 8])
def test_chain_of_calls_matches_oracle(F, cluster):
    """A chain of eight calls with separate bf16 inputs, every cluster size: each output
    against the oracle on its own input."""
    T = 2
    layers = _chain_layers(SMALL_STACK, T, seed=300)
    calls, xs, ys = [], [], []
    for i, ((count, out_f, in_f), lin) in enumerate(zip(SMALL_STACK, layers)):
        x = synth.outlier_activations(1, in_f, seed=500 + i).to(DEV)
        y = [torch.full((1, out_f), float("nan"), device=DEV) for _ in range(count)]
        calls.append((x, [d for _, _, d, _ in lin], [s for _, _, _, s in lin], y, out_f))
        xs.append(x)
        ys.append(y)
    F.wl_matmul_chain(calls, T, cluster_size=cluster)
    assert F.get_status() == 0
    for (count, out_f, in_f), lin, x, y in zip(SMALL_STACK, layers, xs, ys):
        xo = x.float().cpu().numpy()
        for (codes, scales, _, _), yg in zip(lin, y):
            _close(yg.cpu().numpy(), O.wl_matmul(xo, codes, scales, out_f), xo, scales)


def test_chain_consumes_previous_outputs(F):
    """Calls whose input is the previous call's float32 output (and, for the grouped call, one
    member's output feeds the next call): every output buffer starts as NaN, so a call that read
    its input before the previous call finished would not match the oracle evaluated on the
    inputs the GPU actually used."""
    T = 2
    shapes = [(1, 1024, 512), (2, 512, 1024), (1, 300, 512), (3, 1024, 300), (1, 64, 1024)]
    layers = _chain_layers(shapes, T, seed=900)
    x0 = synth.outlier_activations(1, 512, seed=901).float().to(DEV)
    calls, ins, outs = [], [], []
    x = x0
    for (count, out_f, in_f), lin in zip(shapes, layers):
        y = [torch.full((1, out_f), float("nan"), device=DEV) for _ in range(count)]
        calls.append((x, [d for _, _, d, _ in lin], [s for _, _, _, s in lin], y, out_f))
        ins.append(x)
        outs.append(y)
        x = y[-1]            # the next call reads this call's last output
    for cluster in (0, 1, 2):
        for y in outs:
            for t in y:
                t.fill_(float("nan"))
        F.wl_matmul_chain(calls, T, cluster_size=cluster)
        assert F.get_status() == 0
        for (count, out_f, in_f), lin, xin, y in zip(shapes, layers, ins, outs):
            xo = xin.cpu().numpy().astype(np.float64)
            assert np.all(np.isfinite(xo))
            for (codes, scales, _, _), yg in zip(lin, y):
                _close(yg.cpu().numpy(), O.wl_matmul(xo, codes, scales, out_f), xo, scales)


def test_chain_decoder_layer_full_size(F):
    """One LLaMA-2-7B decoder layer's four calls (q/k/v, o, gate/up, down) at full size with the
    bench's weights and activations."""
    T = 2
    calls, refs = [], []
    for gi, names in enumerate((("q", "k", "v"), ("o",), ("gate", "up"), ("down",))):
        shape = {nm: (rows, cols) for nm, rows, cols in synth.PROJECTIONS}
        rows, cols = shape[names[0]]
        cl, sl, yl = [], [], []
        for nm in names:
            pi = [p[0] for p in synth.PROJECTIONS].index(nm)
            seed = synth.weight_seed("stack", 0, pi)
            R = synth.student_t_weight(rows, cols, seed)
            U, W = F.convert(R.to(DEV))
            codes, scales = F.quantize(U, W, T)
            cl.append(codes)
            sl.append(scales)
            yl.append(torch.empty((1, rows), device=DEV))
            refs.append((R, seed, rows, cols, len(calls), len(yl) - 1))
        x = synth.outlier_activations(1, cols, synth.activation_seed(
            synth.weight_seed("stack", 0, [p[0] for p in synth.PROJECTIONS].index(names[0])), 1))
        calls.append((x.to(DEV), cl, sl, yl, rows))
    F.wl_matmul_chain(calls, T)
    assert F.get_status() == 0
    for R, seed, rows, cols, ci, gi in refs[:5]:      # the oracle's time: the first five linears
        Uo, Wo = O.convert(R.numpy())
        co, so = O.quantize(Uo, Wo, T)
        xo = calls[ci][0].float().cpu().numpy()
        _close(calls[ci][3][gi].cpu().numpy(), O.wl_matmul(xo, co, so, rows), xo, so)


def test_chain_repeated_launches_are_deterministic(F):
    T = 2
    layers = _chain_layers(SMALL_STACK[:4], T, seed=77)
    calls = []
    for i, ((count, out_f, in_f), lin) in enumerate(zip(SMALL_STACK[:4], layers)):
        x = synth.outlier_activations(1, in_f, seed=600 + i).to(DEV)
        calls.append((x, [d for _, _, d, _ in lin], [s for _, _, _, s in lin],
                      [torch.empty((1, out_f), device=DEV) for _ in range(count)], out_f))
    ws = F.chain_workspace(len(calls), DEV)
    arr = F.chain_calls(calls)
    F.wl_matmul_chain(None, T, workspace=ws, arr=arr)
    first = [y.clone() for c in calls for y in c[3]]
    for _ in range(3):
        F.wl_matmul_chain(None, T, workspace=ws, arr=arr)
    assert F.get_status() == 0
    for a, c in zip(first, [y for c in calls for y in c[3]]):
        assert torch.equal(a, c)


def test_chain_rejects_outside_its_domain(F):
    n, m, T = 16, 64, 2
    codes, scales = _random_quantized(n, m, T, seed=71)
    codes5, scales5 = _random_quantized(n, m, 5, seed=72)
    with pytest.raises(F.Fairy2iError) as e:     # T = 5
        F.wl_matmul(synth.outlier_activations(1, 2 * m, seed=1).to(DEV), _upload(codes5),
                    torch.from_numpy(scales5).to(DEV), 2 * n, path=PATH)
    assert e.value.code == 1
    m2 = 12288 + 128                             # rows longer than the kernel takes
    codes2, scales2 = _random_quantized(2, m2, 1, seed=73)
    with pytest.raises(F.Fairy2iError) as e:
        F.wl_matmul(torch.zeros((1, 2 * m2), dtype=torch.bfloat16, device=DEV), _upload(codes2),
                    torch.from_numpy(scales2).to(DEV), 4, path=PATH)
    assert e.value.code == 1
    assert F.get_status() == 0


def test_chain_element_bound_for_extreme_x(F):
    """x is held to 2^-28 of the largest |x| of a CTA's slice, so the l1 error of x stays below
    in_features 2^-28 |x|_1 and every output within 1e-4 |x~|_1 sum_t s_t, whatever x is. Worst
    case here: the longest rows, x = (1, tiny, tiny, ...) with the tiny entries just under half a
    unit, every code +1 so that the errors add up, the K split forced to 4 (slices of 6144)."""
    T, out_f, in_f = 2, 2048, 24576
    tiny = 0.99609375 * 2.0**-28
    n, m = O.complex_dims(out_f, in_f)
    codes = np.zeros((T, 2, n, m), dtype=np.uint8)
    scales = np.full((T, 2, 2), 0.02, dtype=np.float32)
    x = torch.full((1, in_f), tiny, dtype=torch.float32).to(torch.bfloat16)
    x[0, 0] = 1.0
    y = torch.empty((1, out_f), device=DEV)
    xd = x.to(DEV)
    F.wl_matmul_chain([(xd, [_upload(codes)], [torch.from_numpy(scales).to(DEV)], [y], out_f)], T,
                      cluster_size=4)
    assert F.get_status() == 0
    xo = x.float().numpy().astype(np.float64)
    err = np.asarray(y.cpu().numpy(), np.float64) - O.wl_matmul(xo, codes, scales, out_f)
    bound = 1e-4 * O.tolerance_bound(xo, scales)[:, None]
    assert np.max(np.abs(err) - bound) <= 0, f"element error {np.max(np.abs(err) / bound):.3f} of the bound"
