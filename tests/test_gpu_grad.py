"""GPU parity of the QAT gradients against the CPU oracle: the straight-through weight gradient
(dU = sum_b g_b conj(x_b)^T, dW = sum_b g_b x_b^T, one real GEMM on the tensor cores) and the
master gradient through the scales of the residual stages.

Tolerances. Weight gradient: bf16 x and g are exact, products exact in the f32 accumulator, the
sums over B tokens rounded in f32: relative Frobenius <= 1e-5 and, per element,
|err| <= 1e-5 sum_b |g_b| |x_b| (the scale of that entry's sum). Scale path: float64 sums, float32
outputs, the residual replayed exactly as the quantizer computes it: relative 1e-6 on the scale
gradients and relative Frobenius 1e-6 on the master gradient."""
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


@pytest.mark.parametrize("B,out_f,in_f", [(1, 8, 8), (7, 31, 515), (64, 128, 128),
                                          (100, 300, 260), (2048, 4096, 4096), (256, 11008, 4096)])
def test_ste_weight_grad_matches_oracle(F, B, out_f, in_f):
    x = synth.outlier_activations(B, in_f, seed=B + in_f)
    g = (torch.randn(B, out_f, generator=torch.Generator().manual_seed(out_f + B)) * 0.1).to(torch.bfloat16)
    dU, dW = F.ste_weight_grad(x.to(DEV), g.to(DEV))
    assert F.get_status() == 0
    n, m = O.complex_dims(out_f, in_f)
    xo, go = x.double().numpy(), g.double().numpy()
    eU, eW = O.ste_weight_grad(xo, go, n, m)
    zabs = np.abs(O.split_input(xo, m))
    gabs = np.abs(O.split_input(go, n))
    scale = gabs.T @ zabs                      # sum_b |g_b| |x_b|
    for got, want in ((dU, eU), (dW, eW)):
        got = got.cpu().numpy().astype(np.complex128)
        assert np.linalg.norm(got - want) <= 1e-5 * np.linalg.norm(want)
        assert np.all(np.abs(got - want) <= 1e-5 * scale + 1e-30)


def test_ste_weight_grad_accumulates(F):
    B, out_f, in_f = 32, 96, 200
    x = synth.outlier_activations(B, in_f, seed=3).to(DEV)
    g = (0.1 * torch.randn(B, out_f, generator=torch.Generator().manual_seed(4))).to(torch.bfloat16).to(DEV)
    dU, dW = F.ste_weight_grad(x, g)
    dU2, dW2 = F.ste_weight_grad(x, g, dU=dU.clone(), dW=dW.clone(), accumulate=True)
    assert F.get_status() == 0
    assert torch.allclose(dU2, 2 * dU, rtol=1e-6, atol=0) and torch.allclose(dW2, 2 * dW, rtol=1e-6, atol=0)


@pytest.mark.parametrize("rows,cols,T", [(64, 64, 1), (130, 258, 2), (512, 1024, 3), (4096, 4096, 2)])
def test_scale_grad_matches_oracle(F, rows, cols, T):
    R = synth.student_t_weight(rows, cols, seed=rows + cols + T)
    U, W = F.convert(R.to(DEV))
    codes, scales = F.quantize(U, W, T)
    n, m = U.shape
    g = torch.Generator().manual_seed(T)
    dU = (torch.randn(n, m, generator=g) + 1j * torch.randn(n, m, generator=g)).to(torch.complex64)
    dW = (torch.randn(n, m, generator=g) + 1j * torch.randn(n, m, generator=g)).to(torch.complex64)
    gU, gW, shat = F.scale_grad(U, W, codes, scales, dU.to(DEV), dW.to(DEV))
    assert F.get_status() == 0
    co = O.unpack_codes(codes.cpu().numpy().view(np.uint32).reshape(-1), T, n, m)
    so = scales.cpu().numpy()
    for M, (Mt, dMt, gMt) in enumerate(((U, dU, gU), (W, dW, gW))):
        want, swant = O.scale_path_grad(Mt.cpu().numpy(), co[:, M], so[:, M], dMt.numpy(),
                                        mode="contract")
        got = gMt.cpu().numpy().astype(np.complex128)
        assert np.linalg.norm(got - want) <= 1e-6 * np.linalg.norm(want)
        sg = shat.cpu().numpy()[:, M]
        assert np.allclose(sg, swant, rtol=1e-6, atol=1e-6 * np.abs(swant).max())
