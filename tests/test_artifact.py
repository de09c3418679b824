"""Save/load of a quantized layer (packed codes + scales): round trip and the checks on load.
CPU only; the library is loaded for its word-count function."""
import numpy as np
import pytest
import torch

from paper_2512_02901_gb300 import artifact, binding


@pytest.fixture(scope="module", autouse=True)
def _built_library():
    import __graft_entry__ as entry
    entry.build()
    binding.load()


def _layer(out_f, in_f, T, seed):
    n, m = (out_f + 1) // 2, (in_f + 1) // 2
    words = int(binding.load().fairy2i_codes_words(n, m, T))
    g = np.random.default_rng(seed)
    codes = torch.from_numpy(g.integers(-2**31, 2**31 - 1, words, dtype=np.int64).astype(np.int32))
    scales = torch.from_numpy((0.01 + 0.02 * g.random((T, 2, 2))).astype(np.float32))
    return codes, scales


@pytest.mark.parametrize("out_f,in_f,T", [(33, 70, 3), (4096, 4096, 2), (1, 1, 1), (9, 300, 8)])
def test_round_trip(tmp_path, out_f, in_f, T):
    codes, scales = _layer(out_f, in_f, T, seed=out_f + in_f + T)
    p = str(tmp_path / "layer.f2i")
    artifact.save(p, codes, scales, out_f, in_f, T)
    c2, s2, o2, i2, t2 = artifact.load(p)
    assert (o2, i2, t2) == (out_f, in_f, T)
    assert c2.dtype == torch.int32 and torch.equal(c2, codes)
    assert s2.shape == (T, 2, 2) and torch.equal(s2, scales)


def test_linear_load_without_weight(tmp_path):
    codes, scales = _layer(100, 64, 2, seed=1)
    p = str(tmp_path / "layer.f2i")
    artifact.save(p, codes, scales, 100, 64, 2)
    layer = binding.Fairy2iLinear.load(p, device="cpu")
    assert (layer.out_features, layer.in_features, layer.T) == (100, 64, 2)
    assert torch.equal(layer.codes, codes) and torch.equal(layer.scales, scales)


def test_save_rejects_wrong_sizes(tmp_path):
    codes, scales = _layer(33, 70, 3, seed=2)
    with pytest.raises(ValueError):
        artifact.save(str(tmp_path / "a"), codes[:-1], scales, 33, 70, 3)
    with pytest.raises(ValueError):
        artifact.save(str(tmp_path / "b"), codes, scales[:2], 33, 70, 3)
    with pytest.raises(ValueError):   # the word count of another shape
        artifact.save(str(tmp_path / "c"), codes, scales, 33, 700, 3)


def test_load_rejects_damaged_files(tmp_path):
    codes, scales = _layer(33, 70, 3, seed=3)
    p = tmp_path / "layer.f2i"
    artifact.save(str(p), codes, scales, 33, 70, 3)
    good = p.read_bytes()
    cases = {
        "magic": b"NOTFAIRY" + good[8:],
        "version": good[:8] + (2).to_bytes(4, "little") + good[12:],
        "shape": good[:16] + (34000).to_bytes(8, "little") + good[24:],
        "truncated": good[:-4],
        "trailing": good + b"\0\0\0\0",
        "header": good[:10],
    }
    for name, data in cases.items():
        q = tmp_path / f"{name}.f2i"
        q.write_bytes(data)
        with pytest.raises(ValueError):
            artifact.load(str(q))
