"""ctypes binding of libfairy2i.so: argument marshalling only. Every step of the path runs in
the library's CUDA kernels; torch provides device memory and streams. There is no CPU
fallback: a missing library raises."""
from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libfairy2i.so")

F32, BF16 = 0, 1
PATH_AUTO, PATH_DECODE, PATH_TC_PREFILL, PATH_STREAM, PATH_CHAIN = 0, 1, 3, 4, 5
MAX_STAGES = 8
STATUS = {0: "ok", 1: "invalid argument", 2: "shape", 3: "alignment", 4: "dtype", 5: "workspace",
          6: "non-finite weight", 7: "device wait timeout", 8: "CUDA error"}

_lib = None

_c = ctypes
_i64, _vp, _int, _sz = _c.c_int64, _c.c_void_p, _c.c_int, _c.c_size_t
SIGNATURES = {
    "fairy2i_status_string": ([_int], _c.c_char_p),
    "fairy2i_convert": ([_vp, _i64, _i64, _i64, _vp, _vp, _i64, _vp], _int),
    "fairy2i_codes_words_per_row": ([_i64], _i64),
    "fairy2i_codes_words": ([_i64, _i64, _int], _i64),
    "fairy2i_quantize_workspace_bytes": ([_i64, _i64, _int], _sz),
    "fairy2i_quantize": ([_vp, _vp, _i64, _i64, _i64, _int, _vp, _vp, _vp, _sz, _vp], _int),
    "fairy2i_wl_matmul": ([_vp, _int, _i64, _i64, _i64, _vp, _vp, _i64, _int, _vp, _i64, _vp],
                          _int),
    "fairy2i_wl_matmul_path": ([_vp, _int, _i64, _i64, _i64, _vp, _vp, _i64, _int, _vp, _i64,
                                _int, _vp], _int),
    "fairy2i_get_status": ([_vp], _int),
    "fairy2i_quantize_noalloc": ([_vp, _vp, _i64, _i64, _i64, _int, _vp, _vp, _vp], _int),
    "fairy2i_selftest_wait_timeout": ([_c.c_uint32, _vp], _int),
    "fairy2i_wl_matmul_group": ([_vp, _int, _i64, _i64, _i64, _int, _vp, _vp, _i64, _int, _vp,
                                 _i64, _vp], _int),
    "fairy2i_codes_adjoint": ([_vp, _i64, _i64, _int, _vp, _vp], _int),
    "fairy2i_wl_matmul_group_path": ([_vp, _int, _i64, _i64, _i64, _int, _vp, _vp, _i64, _int,
                                      _vp, _i64, _int, _vp], _int),
}
MAX_GROUP = 4


class ChainCall(ctypes.Structure):
    """fairy2i_chain_call: one call of a chained decode (one token, up to MAX_GROUP linears)."""
    _fields_ = [("x", _vp), ("xdt", _int), ("count", ctypes.c_int32),
                ("in_features", _i64), ("out_features", _i64),
                ("codes", _vp * 4), ("scales", _vp * 4), ("y", _vp * 4)]


SIGNATURES.update({
    "fairy2i_hermitian_attention_workspace_bytes": ([_i64, _int, _i64], _sz),
    "fairy2i_hermitian_attention": ([_vp, _vp, _vp, _i64, _i64, _i64, _int, _vp, _vp, _sz, _vp],
                                    _int),
    "fairy2i_rmsnorm": ([_vp, _vp, _vp, _i64, _i64, _c.c_float, _vp, _vp, _vp], _int),
    "fairy2i_silu_mul": ([_vp, _vp, _i64, _vp, _vp], _int),
    "fairy2i_lut_quantize_x": ([_vp, _i64, _vp, _vp], _int),
    "fairy2i_lut_workspace_bytes": ([_i64], _sz),
    "fairy2i_lut_matmul": ([_vp, _c.c_float, _i64, _vp, _vp, _i64, _int, _vp, _vp, _sz, _int],
                           _int),
    "fairy2i_ste_weight_grad_workspace_bytes": ([_i64, _i64, _i64], _sz),
    "fairy2i_ste_weight_grad": ([_vp, _i64, _vp, _i64, _i64, _i64, _i64, _vp, _vp, _i64, _int,
                                 _vp, _sz, _vp], _int),
    "fairy2i_scale_grad_workspace_bytes": ([], _sz),
    "fairy2i_scale_grad": ([_vp, _vp, _i64, _i64, _i64, _int, _vp, _vp, _vp, _vp, _i64, _vp, _vp,
                            _i64, _vp, _vp, _sz, _vp], _int),
    "fairy2i_wl_matmul_chain_max_calls": ([], _int),
    "fairy2i_wl_matmul_chain_workspace_bytes": ([_int], _sz),
    "fairy2i_wl_matmul_chain": ([_vp, _int, _int, _int, _vp, _sz, _vp], _int),
})


class Fairy2iError(RuntimeError):
    def __init__(self, call: str, code: int):
        super().__init__(f"{call}: {STATUS.get(code, code)} ({code})")
        self.code = code


def load(path: str = LIB_PATH):
    """Opens the library (once). Raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(path):
            raise RuntimeError(f"libfairy2i.so not built ({path}); run "
                               "paper_2512_02901_gb300.build.build() first")
        lib = ctypes.CDLL(path)
        for name, (args, res) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.argtypes, fn.restype = args, res
        _lib = lib
    return _lib


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check(call: str, code: int):
    if code != 0:
        raise Fairy2iError(call, code)


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr())


def complex_dims(rows: int, cols: int):
    return (rows + 1) // 2, (cols + 1) // 2


def words_per_row(m: int) -> int:
    return int(load().fairy2i_codes_words_per_row(m))


def convert(R: torch.Tensor, stream=None):
    """R float32 [rows][cols] (CUDA, row stride >= cols) -> U, W complex64 [n][m]."""
    assert R.is_cuda and R.dtype == torch.float32 and R.dim() == 2 and R.stride(1) == 1
    rows, cols = R.shape
    n, m = complex_dims(rows, cols)
    U = torch.empty((n, m), dtype=torch.complex64, device=R.device)
    W = torch.empty((n, m), dtype=torch.complex64, device=R.device)
    _check("fairy2i_convert", load().fairy2i_convert(_ptr(R), rows, cols, R.stride(0), _ptr(U),
                                                     _ptr(W), m, _stream(stream)))
    return U, W


def quantize_workspace_bytes(n: int, m: int, T: int) -> int:
    return int(load().fairy2i_quantize_workspace_bytes(n, m, T))


def quantize(U: torch.Tensor, W: torch.Tensor, T: int, codes=None, scales=None, workspace=None,
             stream=None):
    """U, W complex64 [n][m] (CUDA) -> codes: int32 view of the packed uint32 words,
    shape [T][2][ceil(n/16)][wpr/8][16][8]; scales float32 [T][2][2]."""
    assert U.is_cuda and U.dtype == torch.complex64 and U.shape == W.shape and W.dtype == U.dtype
    assert U.stride(1) == 1 and W.stride(0) == U.stride(0) and W.stride(1) == 1
    n, m = U.shape
    wpr = words_per_row(m)
    dev = U.device
    if codes is None:
        codes = torch.empty((T, 2, (n + 15) // 16, wpr // 8, 16, 8), dtype=torch.int32, device=dev)
    if scales is None:
        scales = torch.empty((T, 2, 2), dtype=torch.float32, device=dev)
    nbytes = quantize_workspace_bytes(n, m, T)
    if workspace is None or workspace.numel() < nbytes:
        workspace = torch.empty(max(nbytes, 1), dtype=torch.uint8, device=dev)
    _check("fairy2i_quantize",
           load().fairy2i_quantize(_ptr(torch.view_as_real(U)), _ptr(torch.view_as_real(W)), n, m,
                                   U.stride(0), T, _ptr(codes), _ptr(scales), _ptr(workspace),
                                   workspace.numel(), _stream(stream)))
    return codes, scales


def check_layer(codes: torch.Tensor, scales: torch.Tensor, out_features: int, in_features: int,
                T: int, device=None) -> None:
    """Raises ValueError unless (codes, scales) can hold a T-stage layer of out_features x
    in_features on `device`: the packed words at least fairy2i_codes_words(n, m, T) (int32 or
    uint32, contiguous) and float32 contiguous scales of at least [T][2][2]. A mismatch would let
    a kernel read past the end of the codes buffer, so it is caught before any launch."""
    if not (1 <= T <= MAX_STAGES):
        raise ValueError(f"T = {T} outside 1..{MAX_STAGES}")
    if out_features < 1 or in_features < 1:
        raise ValueError("out_features and in_features must be >= 1")
    n, m = complex_dims(out_features, in_features)
    need = T * 2 * ((n + 15) // 16) * 16 * (((m + 127) // 128) * 8)
    if codes.dtype not in (torch.int32, torch.uint32) or not codes.is_contiguous():
        raise ValueError("codes must be a contiguous int32/uint32 tensor of packed words")
    if codes.numel() < need:
        raise ValueError(f"codes hold {codes.numel()} words, a {T}-stage {out_features}x"
                         f"{in_features} layer needs {need}")
    if scales.dtype != torch.float32 or not scales.is_contiguous() or scales.numel() < 4 * T:
        raise ValueError(f"scales must be contiguous float32 with at least [T][2][2] = {4 * T} "
                         f"values (got {tuple(scales.shape)}, {scales.dtype})")
    if device is not None and (codes.device != device or scales.device != device):
        raise ValueError(f"codes ({codes.device}) and scales ({scales.device}) must be on {device}")


def wl_matmul(x: torch.Tensor, codes: torch.Tensor, scales: torch.Tensor, out_features: int,
              y=None, path: int = PATH_AUTO, stream=None, T: int | None = None):
    """x [B][in_features] float32/bf16 -> y float32 [B][out_features] = [Re y | Im y].
    A CPU x is copied to the device (pinned staging) and y copied back: the end-to-end form."""
    if not x.is_cuda:
        dev = codes.device
        xd = x.pin_memory().to(dev, non_blocking=True) if not x.is_pinned() else x.to(dev, non_blocking=True)
        yd = wl_matmul(xd, codes, scales, out_features, path=path, stream=stream, T=T)
        out = torch.empty(yd.shape, dtype=yd.dtype, pin_memory=True) if y is None else y
        out.copy_(yd, non_blocking=True)
        torch.cuda.current_stream(dev).synchronize() if stream is None else stream.synchronize()
        return out
    assert x.dim() == 2 and x.stride(1) == 1 and x.dtype in (torch.float32, torch.bfloat16)
    B, in_features = x.shape
    if T is None:
        T = scales.shape[0]
    check_layer(codes, scales, out_features, in_features, T, x.device)
    if y is None:
        y = torch.empty((B, out_features), dtype=torch.float32, device=x.device)
    assert y.is_cuda and y.dtype == torch.float32 and y.stride(1) == 1 and \
        y.shape[0] >= B and y.shape[1] >= out_features
    xdt = F32 if x.dtype == torch.float32 else BF16
    _check("fairy2i_wl_matmul",
           load().fairy2i_wl_matmul_path(_ptr(x), xdt, B, in_features, x.stride(0), _ptr(codes),
                                         _ptr(scales), out_features, T, _ptr(y), y.stride(0),
                                         path, _stream(stream)))
    return y


def wl_matmul_group(x: torch.Tensor, codes, scales, out_features: int, ys=None, stream=None,
                    T: int | None = None, path: int = PATH_AUTO):
    """Several linears of the same shape on one input x (CUDA): returns [y_g] with
    y_g = wl_matmul(x, codes[g], scales[g], out_features); one launch where a decode kernel
    applies (path 0 automatic, 1 the warp-MMA decode kernel, 3 the tcgen05 prefill GEMM at any B,
    4 the persistent tcgen05 decode kernel, 5 the chained one)."""
    assert x.is_cuda and x.dim() == 2 and x.stride(1) == 1 and x.dtype in (torch.float32,
                                                                          torch.bfloat16)
    count = len(codes)
    assert count == len(scales) and 1 <= count <= MAX_GROUP
    B, in_features = x.shape
    if T is None:
        T = scales[0].shape[0]
    for c, s in zip(codes, scales):
        check_layer(c, s, out_features, in_features, T, x.device)
    if ys is None:
        ys = [torch.empty((B, out_features), dtype=torch.float32, device=x.device)
              for _ in range(count)]
    assert len(ys) == count and all(y.stride(0) == ys[0].stride(0) for y in ys)
    assert all(y.is_cuda and y.dtype == torch.float32 and y.stride(1) == 1 and
               y.shape[0] >= B and y.shape[1] >= out_features for y in ys)
    arr = ctypes.c_void_p * count
    cp = arr(*[c.data_ptr() for c in codes])
    sp = arr(*[s.data_ptr() for s in scales])
    yp = arr(*[y.data_ptr() for y in ys])
    xdt = F32 if x.dtype == torch.float32 else BF16
    _check("fairy2i_wl_matmul_group_path",
           load().fairy2i_wl_matmul_group_path(_ptr(x), xdt, B, in_features, x.stride(0), count,
                                               ctypes.cast(cp, _vp), ctypes.cast(sp, _vp),
                                               out_features, T, ctypes.cast(yp, _vp),
                                               ys[0].stride(0), path, _stream(stream)))
    return ys


def chain_workspace(ncalls: int, device) -> torch.Tensor:
    """Device workspace (completion counters) for a chain of ncalls calls."""
    nbytes = int(load().fairy2i_wl_matmul_chain_workspace_bytes(ncalls))
    return torch.empty(max(nbytes, 16), dtype=torch.uint8, device=device)


def chain_calls(calls):
    """ctypes array of fairy2i_chain_call from (x, codes list, scales list, y list, out_features)
    tuples; x is one token [1][in_features] (float32 or bf16, CUDA), y [1][out_features] float32.
    The layers are checked like wl_matmul's."""
    arr = (ChainCall * len(calls))()
    T = None
    for i, (x, codes, scales, ys, out_features) in enumerate(calls):
        assert x.is_cuda and x.dim() == 2 and x.shape[0] == 1 and x.is_contiguous()
        assert x.dtype in (torch.float32, torch.bfloat16)
        count = len(codes)
        assert count == len(scales) == len(ys) and 1 <= count <= MAX_GROUP
        in_features = x.shape[1]
        if T is None:
            T = scales[0].shape[0]
        for c, s, y in zip(codes, scales, ys):
            check_layer(c, s, out_features, in_features, T, x.device)
            assert y.is_cuda and y.dtype == torch.float32 and y.is_contiguous() and \
                y.numel() >= out_features
        k = arr[i]
        k.x = x.data_ptr()
        k.xdt = F32 if x.dtype == torch.float32 else BF16
        k.count = count
        k.in_features, k.out_features = in_features, out_features
        for g in range(count):
            k.codes[g] = codes[g].data_ptr()
            k.scales[g] = scales[g].data_ptr()
            k.y[g] = ys[g].data_ptr()
    return arr


def wl_matmul_chain(calls, T: int, cluster_size: int = 0, workspace=None, stream=None,
                    arr=None):
    """Runs a chain of one-token calls in one launch (fairy2i_wl_matmul_chain): call c reads its
    x only after every y of call c - 1 is written. `calls`: (x, codes, scales, ys, out_features)
    tuples (see chain_calls), or None with `arr` a prepared chain_calls() array."""
    if arr is None:
        arr = chain_calls(calls)
    n = len(arr)
    if workspace is None:
        dev = torch.device("cuda", torch.cuda.current_device()) if calls is None else \
            calls[0][0].device
        workspace = chain_workspace(n, dev)
    _check("fairy2i_wl_matmul_chain",
           load().fairy2i_wl_matmul_chain(ctypes.cast(arr, _vp), n, T, cluster_size,
                                          _ptr(workspace), workspace.numel(), _stream(stream)))
    return arr


def hermitian_attention(q: torch.Tensor, k_cache: torch.Tensor, v_cache: torch.Tensor, L: int,
                        heads: int, out=None, workspace=None, stream=None) -> torch.Tensor:
    """Attention of one query over the first L cached positions with Hermitian scores
    (fairy2i_hermitian_attention). q float32 [2 n] ([Re | Im]); caches float32 [Lmax][2 n]
    (rows as wl_matmul writes them); returns float32 [2 n]."""
    assert q.is_cuda and q.dtype == torch.float32 and q.is_contiguous()
    for c in (k_cache, v_cache):
        assert c.is_cuda and c.dtype == torch.float32 and c.dim() == 2 and c.stride(1) == 1
        assert c.shape[0] >= L and c.shape[1] >= q.numel()
    n = q.numel() // 2
    if out is None:
        out = torch.empty(2 * n, dtype=torch.float32, device=q.device)
    nbytes = int(load().fairy2i_hermitian_attention_workspace_bytes(n, heads, L))
    if workspace is None or workspace.numel() < nbytes:
        workspace = torch.empty(max(nbytes, 4), dtype=torch.uint8, device=q.device)
    _check("fairy2i_hermitian_attention",
           load().fairy2i_hermitian_attention(_ptr(q), _ptr(k_cache), _ptr(v_cache), L,
                                              k_cache.stride(0), n, heads, _ptr(out),
                                              _ptr(workspace), workspace.numel(), _stream(stream)))
    return out


def rmsnorm(h: torch.Tensor, w: torch.Tensor, eps: float, delta=None, h_out=None, out=None,
            stream=None) -> torch.Tensor:
    """out = (h + delta) / sqrt(mean((h + delta)^2) + eps) * w per token (fairy2i_rmsnorm);
    h_out, if given, receives h + delta. h [B][d] float32 (CUDA)."""
    assert h.is_cuda and h.dtype == torch.float32 and h.is_contiguous()
    h2 = h.view(-1, h.shape[-1])
    B, d = h2.shape
    assert w.numel() == d and w.dtype == torch.float32 and w.is_contiguous()
    if delta is not None:
        assert delta.shape == h.shape and delta.dtype == torch.float32 and delta.is_contiguous()
    if out is None:
        out = torch.empty_like(h)
    _check("fairy2i_rmsnorm",
           load().fairy2i_rmsnorm(_ptr(h), _ptr(delta) if delta is not None else None, _ptr(w), B,
                                  d, eps, _ptr(h_out) if h_out is not None else None, _ptr(out),
                                  _stream(stream)))
    return out


def silu_mul(g: torch.Tensor, u: torch.Tensor, out=None, stream=None) -> torch.Tensor:
    """silu(g) * u elementwise (fairy2i_silu_mul), float32 CUDA tensors of the same size."""
    assert g.is_cuda and g.dtype == torch.float32 and g.is_contiguous() and u.shape == g.shape
    if out is None:
        out = torch.empty_like(g)
    _check("fairy2i_silu_mul", load().fairy2i_silu_mul(_ptr(g), _ptr(u), g.numel(), _ptr(out),
                                                       _stream(stream)))
    return out


def lut_quantize_x(x: torch.Tensor):
    """int8 activations of one token on the host (fairy2i_lut_quantize_x): returns (xq, delta)."""
    x = x.detach().to("cpu", torch.float32).contiguous().view(-1)
    xq = torch.empty(x.numel(), dtype=torch.int8)
    sc = ctypes.c_float()
    _check("fairy2i_lut_quantize_x",
           load().fairy2i_lut_quantize_x(_ptr(x), x.numel(), _ptr(xq), ctypes.byref(sc)))
    return xq, float(sc.value)


def lut_matmul(xq: torch.Tensor, delta: float, codes: torch.Tensor, scales: torch.Tensor,
               out_features: int, T: int | None = None, nthreads: int | None = None,
               workspace=None) -> torch.Tensor:
    """The host look-up-table matmul (fairy2i_lut_matmul) of one int8 token: host tensors."""
    assert xq.dtype == torch.int8 and not xq.is_cuda and xq.is_contiguous()
    codes = codes.detach().to("cpu").contiguous()
    scales = scales.detach().to("cpu", torch.float32).contiguous()
    in_features = xq.numel()
    if T is None:
        T = scales.shape[0]
    check_layer(codes, scales, out_features, in_features, T)
    nbytes = int(load().fairy2i_lut_workspace_bytes(in_features))
    if workspace is None or workspace.numel() < nbytes:
        workspace = torch.empty(nbytes, dtype=torch.uint8)
    y = torch.empty(out_features, dtype=torch.float32)
    nthreads = nthreads or (os.cpu_count() or 1)
    _check("fairy2i_lut_matmul",
           load().fairy2i_lut_matmul(_ptr(xq), delta, in_features, _ptr(codes), _ptr(scales),
                                     out_features, T, _ptr(y), _ptr(workspace), workspace.numel(),
                                     nthreads))
    return y


def ste_weight_grad(x: torch.Tensor, g: torch.Tensor, dU=None, dW=None, accumulate: bool = False,
                    stream=None):
    """dL/dU^, dL/dW^ (complex64 [n][m]) of a layer from its bf16 input x [B][in] and output
    gradient g [B][out] (fairy2i_ste_weight_grad); added to dU, dW when accumulate."""
    assert x.is_cuda and g.is_cuda and x.dtype == torch.bfloat16 and g.dtype == torch.bfloat16
    assert x.dim() == 2 and g.dim() == 2 and x.shape[0] == g.shape[0]
    assert x.stride(1) == 1 and g.stride(1) == 1
    B, in_f = x.shape
    out_f = g.shape[1]
    n, m = complex_dims(out_f, in_f)
    if dU is None:
        dU = torch.zeros((n, m), dtype=torch.complex64, device=x.device)
    if dW is None:
        dW = torch.zeros((n, m), dtype=torch.complex64, device=x.device)
    assert dU.shape == (n, m) and dW.shape == (n, m) and dU.is_contiguous() and dW.is_contiguous()
    nb = int(load().fairy2i_ste_weight_grad_workspace_bytes(B, in_f, out_f))
    ws = torch.empty(nb, dtype=torch.uint8, device=x.device)
    _check("fairy2i_ste_weight_grad",
           load().fairy2i_ste_weight_grad(_ptr(x), x.stride(0), _ptr(g), g.stride(0), B, in_f,
                                          out_f, _ptr(torch.view_as_real(dU)),
                                          _ptr(torch.view_as_real(dW)), m, int(accumulate),
                                          _ptr(ws), nb, _stream(stream)))
    return dU, dW


def scale_grad(U: torch.Tensor, W: torch.Tensor, codes: torch.Tensor, scales: torch.Tensor,
               dU: torch.Tensor, dW: torch.Tensor, T: int | None = None, stream=None):
    """Master gradient through the scales (fairy2i_scale_grad): returns (gU, gW, shat) with
    gU, gW complex64 [n][m] and shat float32 [T][2][2]."""
    n, m = U.shape
    if T is None:
        T = scales.shape[0]
    for t in (U, W, dU, dW):
        assert t.is_cuda and t.dtype == torch.complex64 and t.shape == (n, m) and t.is_contiguous()
    gU = torch.empty_like(U)
    gW = torch.empty_like(W)
    shat = torch.empty((T, 2, 2), dtype=torch.float32, device=U.device)
    nb = int(load().fairy2i_scale_grad_workspace_bytes())
    ws = torch.empty(nb, dtype=torch.uint8, device=U.device)
    r = torch.view_as_real
    _check("fairy2i_scale_grad",
           load().fairy2i_scale_grad(_ptr(r(U)), _ptr(r(W)), n, m, m, T, _ptr(codes), _ptr(scales),
                                     _ptr(r(dU)), _ptr(r(dW)), m, _ptr(r(gU)), _ptr(r(gW)), m,
                                     _ptr(shat), _ptr(ws), nb, _stream(stream)))
    return gU, gW, shat


def codes_adjoint(codes: torch.Tensor, n: int, m: int, T: int, stream=None) -> torch.Tensor:
    """Codes of the adjoint layer (input gradient, R^T): the layout fairy2i_quantize writes for
    an m x n layer. wl_matmul(y_grad, codes_adjoint(...), scales, in_features) = x~_grad."""
    out = torch.empty(int(load().fairy2i_codes_words(m, n, T)), dtype=torch.int32,
                      device=codes.device)
    _check("fairy2i_codes_adjoint",
           load().fairy2i_codes_adjoint(_ptr(codes), n, m, T, _ptr(out), _stream(stream)))
    return out


def selftest_wait_timeout(limit_us: int, stream=None):
    """Runs the device-side bounded wait on a barrier nothing completes (gives up after about
    limit_us microseconds and latches the timeout status; read it with get_status)."""
    _check("fairy2i_selftest_wait_timeout",
           load().fairy2i_selftest_wait_timeout(limit_us, _stream(stream)))


def get_status(stream=None) -> int:
    """Synchronizes the stream and returns (and clears) the device-side status code."""
    return int(load().fairy2i_get_status(_stream(stream)))


class Fairy2iLinear:
    """A real linear layer (weight [out][in], fp32) converted and quantized once; calls run the
    quantized widely-linear matmul."""

    def __init__(self, weight: torch.Tensor, T: int = 2):
        self.out_features, self.in_features = weight.shape
        self.T = T
        U, W = convert(weight)
        self.codes, self.scales = quantize(U, W, T)

    def __call__(self, x: torch.Tensor, path: int = PATH_AUTO) -> torch.Tensor:
        return wl_matmul(x, self.codes, self.scales, self.out_features, path=path)

    def save(self, path: str) -> None:
        """Writes the packed codes and scales (see artifact.py for the format)."""
        from . import artifact
        artifact.save(path, self.codes, self.scales, self.out_features, self.in_features, self.T)

    @classmethod
    def load(cls, path: str, device="cuda") -> "Fairy2iLinear":
        """A layer from a file written by save(), without the original weight."""
        from . import artifact
        layer = cls.__new__(cls)
        layer.codes, layer.scales, layer.out_features, layer.in_features, layer.T = \
            artifact.load(path, device)
        return layer


class WLDecoderLayer:
    """A decoder layer whose seven linears are quantized widely-linear maps and whose attention
    uses Hermitian scores (Sec. 3.1), for one token at a time with a key/value cache. Every step
    is a library call on the device: RMS norm (with the residual add of the previous sub-layer
    fused in), the grouped q/k/v matmul writing the new key and value straight into the caches,
    attention, o, gate/up, silu * up, down. Activations are float32 (the chained decode kernel).

    step(h, delta) takes the residual stream as h + delta and returns (h1, d) with the layer's
    output h1 + d, so the next layer (or a final norm) fuses that add too."""

    NAMES = ("q", "k", "v", "o", "gate", "up", "down")

    def __init__(self, weights: dict, w_attn: torch.Tensor, w_mlp: torch.Tensor, heads: int,
                 max_len: int, T: int = 2, eps: float = 1e-5):
        self.d = weights["q"].shape[1]
        self.dff = weights["gate"].shape[0]
        self.heads, self.T, self.eps, self.max_len = heads, T, eps, max_len
        dev = weights["q"].device
        self.codes, self.scales = {}, {}
        for nm in self.NAMES:
            U, W = convert(weights[nm])
            self.codes[nm], self.scales[nm] = quantize(U, W, T)
        self.w_attn, self.w_mlp = w_attn.contiguous(), w_mlp.contiguous()
        self.k_cache = torch.zeros((max_len, self.d), dtype=torch.float32, device=dev)
        self.v_cache = torch.zeros((max_len, self.d), dtype=torch.float32, device=dev)
        self.pos = 0
        f = lambda *s: torch.empty(s, dtype=torch.float32, device=dev)
        self.x, self.q, self.a, self.o = f(1, self.d), f(1, self.d), f(1, self.d), f(1, self.d)
        self.h1, self.x2 = f(1, self.d), f(1, self.d)
        self.g, self.u, self.m = f(1, self.dff), f(1, self.dff), f(1, self.dff)
        self.dn = f(1, self.d)
        self.ws = torch.empty(max(int(load().fairy2i_hermitian_attention_workspace_bytes(
            self.d // 2, heads, max_len)), 4), dtype=torch.uint8, device=dev)

    def step(self, h: torch.Tensor, delta=None, stream=None):
        assert self.pos < self.max_len
        p = self.pos
        rmsnorm(h, self.w_attn, self.eps, delta=delta, h_out=h if delta is not None else None,
                out=self.x, stream=stream)
        wl_matmul_group(self.x, [self.codes[n] for n in ("q", "k", "v")],
                        [self.scales[n] for n in ("q", "k", "v")], self.d,
                        ys=[self.q, self.k_cache[p:p + 1], self.v_cache[p:p + 1]],
                        path=PATH_CHAIN, stream=stream, T=self.T)
        hermitian_attention(self.q.view(-1), self.k_cache, self.v_cache, p + 1, self.heads,
                            out=self.a.view(-1), workspace=self.ws, stream=stream)
        wl_matmul(self.a, self.codes["o"], self.scales["o"], self.d, y=self.o, path=PATH_CHAIN,
                  stream=stream, T=self.T)
        rmsnorm(h, self.w_mlp, self.eps, delta=self.o, h_out=self.h1, out=self.x2, stream=stream)
        wl_matmul_group(self.x2, [self.codes["gate"], self.codes["up"]],
                        [self.scales["gate"], self.scales["up"]], self.dff, ys=[self.g, self.u],
                        path=PATH_CHAIN, stream=stream, T=self.T)
        silu_mul(self.g, self.u, out=self.m, stream=stream)
        wl_matmul(self.m, self.codes["down"], self.scales["down"], self.d, y=self.dn,
                  path=PATH_CHAIN, stream=stream, T=self.T)
        self.pos += 1
        return self.h1, self.dn
