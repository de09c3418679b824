"""GPU parity on the LLaMA-2-7B linear stack the bench runs (32 layers x q, k, v, o, gate, up,
down; Student-t weights drawn on the GPU with the per-layer seeds; T = 2): for every one of the
224 linears, codes and scales bit for bit and the B = 1 output within tolerance; for layers 0 and
31 the B = 8 output in full and the B = 64 output on sampled rows. The weights are drawn once and
the same array goes to the library and (copied to the host) to the oracle, which runs in a
spawn-started process pool."""
import multiprocessing as mp
import os

import numpy as np
import pytest
import torch

import oracle as O
from paper_2512_02901_gb300 import synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
T = 2
LAYERS = 32


def _oracle_linear(task):
    """Worker: oracle convert + quantize of one linear and its outputs on the given inputs."""
    R, xs, rows_sample = task
    rows = R.shape[0]
    U, W = O.convert(R)
    codes, scales = O.quantize(U, W, T)
    outs = []
    for x in xs:
        if rows_sample is None:
            outs.append(O.wl_matmul(x, codes, scales, rows))
        else:
            m = codes.shape[3]
            yc = O.wl_matmul_rows(O.split_input(x, m), codes, scales, rows_sample)
            outs.append(np.concatenate([yc.real, yc.imag], axis=1))
    return O.pack_codes(codes), scales, outs


@pytest.fixture(scope="module")
def pool():
    ctx = mp.get_context("spawn")
    p = ctx.Pool(max(1, min(16, (os.cpu_count() or 2) - 1)))
    yield p
    p.close()
    p.join()


@pytest.fixture(scope="module")
def F():
    import __graft_entry__ as entry
    entry.build()
    from paper_2512_02901_gb300 import binding
    binding.load()
    return binding


def _close(yg, yo, x, scales, what):
    yg = np.asarray(yg, np.float64)
    err = yg - yo
    rel = np.linalg.norm(err) / np.linalg.norm(yo)
    assert rel <= 1e-5, f"{what}: relative Frobenius error {rel:.3e}"
    bound = 1e-4 * O.tolerance_bound(np.asarray(x, np.float64), scales)[:, None]
    assert np.all(np.abs(err) <= bound), f"{what}: element error above the bound"


def _gpu_linear(F, L, pi, rows, cols):
    seed = synth.weight_seed("stack", L, pi)
    R = synth.student_t_weight(rows, cols, seed, device=DEV)
    U, W = F.convert(R)
    codes, scales = F.quantize(U, W, T)
    return seed, R, codes, scales


def test_stack_all_linears_codes_scales_and_batch_1(F, pool):
    pending = []
    for L in range(LAYERS):
        for pi, (name, rows, cols) in enumerate(synth.PROJECTIONS):
            seed, R, codes, scales = _gpu_linear(F, L, pi, rows, cols)
            x = synth.outlier_activations(1, cols, synth.activation_seed(seed, 1))
            y = F.wl_matmul(x.to(DEV), codes, scales, rows)
            assert F.get_status() == 0
            task = (R.cpu().numpy(), [x.float().numpy()], None)
            pending.append(((L, name), codes.cpu().numpy().view(np.uint32).reshape(-1),
                            scales.cpu().numpy(), y.cpu().numpy(), x.float().numpy(),
                            pool.apply_async(_oracle_linear, (task,))))
            del R, codes, scales, y
        # collect the finished layers as we go (bounded host memory)
        while len(pending) > 3 * len(synth.PROJECTIONS):
            _check_one(pending.pop(0))
    while pending:
        _check_one(pending.pop(0))


def _check_one(item):
    (L, name), codes_g, scales_g, y_g, x, res = item
    codes_o, scales_o, (y_o,) = res.get(timeout=1200)
    assert np.array_equal(codes_g, codes_o.reshape(-1)), f"codes differ: layer {L} {name}"
    assert np.array_equal(scales_g.view(np.uint32), scales_o.view(np.uint32)), \
        f"scales differ: layer {L} {name}"
    _close(y_g, y_o, x, scales_o, f"layer {L} {name} B=1")


@pytest.mark.parametrize("L", [0, LAYERS - 1])
def test_stack_layer_batches_8_and_64(F, pool, L):
    g = np.random.default_rng(L)
    jobs = []
    for pi, (name, rows, cols) in enumerate(synth.PROJECTIONS):
        seed, R, codes, scales = _gpu_linear(F, L, pi, rows, cols)
        x8 = synth.outlier_activations(8, cols, synth.activation_seed(seed, 8))
        x64 = synth.outlier_activations(64, cols, synth.activation_seed(seed, 64))
        y8 = F.wl_matmul(x8.to(DEV), codes, scales, rows).cpu().numpy()
        y64 = F.wl_matmul(x64.to(DEV), codes, scales, rows).cpu().numpy()
        assert F.get_status() == 0
        n = (rows + 1) // 2
        rws = np.sort(g.choice(n, 64, replace=False))
        full = pool.apply_async(_oracle_linear, ((R.cpu().numpy(), [x8.float().numpy()], None),))
        samp = pool.apply_async(_oracle_linear, ((R.cpu().numpy(), [x64.float().numpy()], rws),))
        jobs.append((name, y8, y64, n, rws, x8.float().numpy(), x64.float().numpy(), full, samp))
        del R, codes, scales
    for name, y8, y64, n, rws, x8, x64, full, samp in jobs:
        _, scales_o, (yo8,) = full.get(timeout=1200)
        _close(y8, yo8, x8, scales_o, f"layer {L} {name} B=8")
        _, _, (yo64,) = samp.get(timeout=1200)
        ys = np.concatenate([y64[:, rws], y64[:, n + rws]], axis=1)
        _close(ys, yo64, x64, scales_o, f"layer {L} {name} B=64 (sampled rows)")
