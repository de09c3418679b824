"""Save and load a quantized layer: its packed codes and scales are the deployable artifact
(2 bits per complex weight and 4 floats per stage, Sec. 3.4 storage); nothing else is needed to
run fairy2i_wl_matmul.

File format (little-endian, no padding):
    8 bytes   magic b"FAIRY2I\\0"
    u32       format version (1)
    u32       T, the number of stages
    i64       out_features, i64 in_features (the real linear's shape)
    i64       number of code words N = fairy2i_codes_words(n, m, T)
    f32[4 T]  scales [T][2][2] = (s_re, s_im) per (stage, U/W)
    u32[N]    packed codes in the library's layout
Loading checks the magic, the version, T and the shape against the word count the library
computes for that shape, and the file length."""
from __future__ import annotations

import os
import struct

import numpy as np
import torch

from . import binding

MAGIC = b"FAIRY2I\0"
VERSION = 1
_HEADER = struct.Struct("<8sIIqqq")


def _words(out_features: int, in_features: int, T: int) -> int:
    n, m = (out_features + 1) // 2, (in_features + 1) // 2
    return int(binding.load().fairy2i_codes_words(n, m, T))


def save(path: str, codes: torch.Tensor, scales: torch.Tensor, out_features: int,
         in_features: int, T: int) -> None:
    """Writes the layer's codes (int32/uint32 words, any device) and scales ([T][2][2] float32)."""
    words = _words(out_features, in_features, T)
    if words < 1:
        raise ValueError(f"no code layout for shape ({out_features}, {in_features}), T = {T}")
    c = codes.detach().reshape(-1).cpu().numpy().view(np.uint32)
    s = scales.detach().reshape(-1).cpu().numpy().astype("<f4", copy=False)
    if c.size != words:
        raise ValueError(f"codes hold {c.size} words, the shape needs {words}")
    if s.size != 4 * T:
        raise ValueError(f"scales hold {s.size} values, T = {T} needs {4 * T}")
    tmp = f"{path}.tmp{os.getpid()}"
    with open(tmp, "wb") as f:
        f.write(_HEADER.pack(MAGIC, VERSION, T, out_features, in_features, words))
        f.write(s.astype("<f4").tobytes())
        f.write(c.astype("<u4").tobytes())
    os.replace(tmp, path)


def load(path: str, device="cpu"):
    """Reads a layer written by save(): returns (codes int32, scales float32 [T][2][2],
    out_features, in_features, T), the tensors on `device`."""
    with open(path, "rb") as f:
        head = f.read(_HEADER.size)
        if len(head) != _HEADER.size:
            raise ValueError(f"{path}: shorter than the header")
        magic, version, T, out_f, in_f, words = _HEADER.unpack(head)
        if magic != MAGIC:
            raise ValueError(f"{path}: not a quantized-layer file")
        if version != VERSION:
            raise ValueError(f"{path}: format version {version}, expected {VERSION}")
        if not (1 <= T <= 8) or out_f < 1 or in_f < 1 or words != _words(out_f, in_f, T):
            raise ValueError(f"{path}: inconsistent header (T {T}, shape ({out_f}, {in_f}), "
                             f"{words} words)")
        body = f.read()
    if len(body) != 16 * T + 4 * words:
        raise ValueError(f"{path}: {len(body)} bytes after the header, expected {16 * T + 4 * words}")
    scales = np.frombuffer(body, dtype="<f4", count=4 * T).reshape(T, 2, 2).astype(np.float32)
    codes = np.frombuffer(body, dtype="<u4", offset=16 * T, count=words).view(np.int32)
    return (torch.from_numpy(codes.copy()).to(device), torch.from_numpy(scales.copy()).to(device),
            out_f, in_f, T)
