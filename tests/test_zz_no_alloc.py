"""fairy2i_quantize_noalloc: the quantizer for callers that cannot allocate device memory at
the call (its scratch is a fixed 4 MiB device array inside the library). Through the C ABI,
two calls in a row must reproduce what fairy2i_quantize (caller-provided workspace) writes,
bit for bit, like every other quantizer comparison here. Kept in a file collected last."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2512_02901_gb300 import synth


@pytest.fixture(scope="module")
def F():
    import __graft_entry__ as entry
    entry.build()
    from paper_2512_02901_gb300 import binding
    binding.load()
    return binding


def _noalloc(F, U, W, T):
    n, m = U.shape
    words = int(F.load().fairy2i_codes_words(n, m, T))
    codes = torch.full((words,), -1, dtype=torch.int32, device=U.device)
    scales = torch.full((T, 2, 2), -1.0, dtype=torch.float32, device=U.device)
    st = F.load().fairy2i_quantize_noalloc(
        ctypes.c_void_p(torch.view_as_real(U).data_ptr()),
        ctypes.c_void_p(torch.view_as_real(W).data_ptr()), n, m, U.stride(0), T,
        ctypes.c_void_p(codes.data_ptr()), ctypes.c_void_p(scales.data_ptr()),
        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 0
    return codes, scales


@pytest.mark.gpu
def test_noalloc_matches_workspace_quantizer_twice(F):
    dev = "cuda:0"
    cases = [(4096, 4096, 2, synth.weight_seed("attn")), (301, 77, 3, 17)]
    for rows, cols, T, seed in cases:
        R = synth.student_t_weight(rows, cols, seed).to(dev)
        U, W = F.convert(R)
        ref_codes, ref_scales = F.quantize(U, W, T)
        for _ in range(2):                         # two calls in a row share the scratch
            codes, scales = _noalloc(F, U, W, T)
            assert F.get_status() == 0
            assert torch.equal(codes, ref_codes.reshape(-1))
            assert torch.equal(scales.view(torch.int32), ref_scales.view(torch.int32))


def test_noalloc_rejects_sizes_beyond_scratch(F):
    P = ctypes.c_void_p(1 << 20)
    lib = F.load()
    # 4096 x 4078 = 16,703,488 complex weights: just beyond the 4 MiB scratch (16,703,232 fit)
    assert lib.fairy2i_quantize_noalloc(P, P, 4096, 4078, 4078, 2, P, P, None) == 5
    assert lib.fairy2i_quantize_noalloc(P, P, 8, 8, 8, 0, P, P, None) == 1
