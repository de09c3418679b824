"""Host-side checks of the Python binding (no GPU): a codes or scales tensor that cannot hold the
layer the call names is rejected before anything reaches the library, so a caller's mistake
(wrong out_features, T taken from another layer's scales) never makes a kernel read past the
codes buffer."""
import pytest
import torch

from paper_2512_02901_gb300 import binding as F


def _words(out_f, in_f, T):
    n, m = F.complex_dims(out_f, in_f)
    return T * 2 * ((n + 15) // 16) * 16 * (((m + 127) // 128) * 8)


def _layer(out_f, in_f, T):
    return (torch.zeros(_words(out_f, in_f, T), dtype=torch.int32),
            torch.zeros((T, 2, 2), dtype=torch.float32))


def test_matching_layer_passes():
    codes, scales = _layer(4096, 4096, 2)
    F.check_layer(codes, scales, 4096, 4096, 2)
    F.check_layer(codes, scales, 4096, 4096, 1)     # a prefix of the stages is a valid layer


@pytest.mark.parametrize("out_f,in_f,T", [(4097, 4096, 2), (4096, 4225, 2), (4096, 4096, 3),
                                          (11008, 4096, 2)])
def test_codes_too_small_for_the_named_layer(out_f, in_f, T):
    codes, scales = _layer(4096, 4096, 2)
    scales = torch.zeros((T, 2, 2), dtype=torch.float32)
    with pytest.raises(ValueError, match="codes hold"):
        F.check_layer(codes, scales, out_f, in_f, T)


def test_scales_too_few_stages():
    codes, _ = _layer(64, 64, 3)
    with pytest.raises(ValueError, match="scales"):
        F.check_layer(codes, torch.zeros((2, 2, 2)), 64, 64, 3)


@pytest.mark.parametrize("bad", ["dtype", "strided", "scale_dtype"])
def test_wrong_dtype_or_layout(bad):
    codes, scales = _layer(64, 64, 2)
    if bad == "dtype":
        codes = codes.to(torch.int64)
    elif bad == "strided":
        codes = torch.zeros(2 * codes.numel(), dtype=torch.int32)[::2]
    else:
        scales = scales.double()
    with pytest.raises(ValueError):
        F.check_layer(codes, scales, 64, 64, 2)


@pytest.mark.parametrize("T", [0, 9])
def test_stage_count_out_of_range(T):
    codes, scales = _layer(64, 64, 2)
    with pytest.raises(ValueError, match="T ="):
        F.check_layer(codes, scales, 64, 64, T)


def test_device_mismatch():
    codes, scales = _layer(64, 64, 2)
    with pytest.raises(ValueError, match="must be on"):
        F.check_layer(codes, scales, 64, 64, 2, torch.device("meta"))
