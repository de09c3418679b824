"""The C-ABI library builds, loads and exports every symbol its header declares; host-side
argument validation returns its errors synchronously (no GPU needed: nothing is enqueued)."""
import ctypes
import os
import re

import pytest

import __graft_entry__ as entry
from paper_2512_02901_gb300 import binding as F

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "fairy2i.h")


@pytest.fixture(scope="module")
def lib():
    entry.build()
    return F.load()


def declared_functions():
    with open(HEADER) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(fairy2i_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_three_calls():
    names = declared_functions()
    for n in ("fairy2i_convert", "fairy2i_quantize", "fairy2i_wl_matmul", "fairy2i_get_status"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
        assert name in F.SIGNATURES, f"binding lacks a signature for {name}"


def test_status_strings(lib):
    for code in range(9):
        assert lib.fairy2i_status_string(code)


def test_size_queries(lib):
    assert lib.fairy2i_codes_words_per_row(1) == 8
    assert lib.fairy2i_codes_words_per_row(128) == 8
    assert lib.fairy2i_codes_words_per_row(129) == 16
    assert lib.fairy2i_codes_words_per_row(5504) == 344
    assert lib.fairy2i_codes_words(5504, 2048, 2) == 2 * 2 * 5504 * 128
    assert lib.fairy2i_codes_words(17, 1, 1) == 2 * 32 * 8
    assert lib.fairy2i_codes_words_per_row(0) == 0
    assert lib.fairy2i_quantize_workspace_bytes(2048, 2048, 2) > 0
    assert lib.fairy2i_quantize_workspace_bytes(2048, 2048, 0) == 0
    assert lib.fairy2i_quantize_workspace_bytes(2048, 2048, 9) == 0


P = ctypes.c_void_p
GOOD = P(1 << 20)            # a 16-byte aligned non-null stand-in; never dereferenced
ODD = P((1 << 20) + 4)


def test_convert_validation(lib):
    assert lib.fairy2i_convert(None, 4, 4, 4, GOOD, GOOD, 2, None) == 1
    assert lib.fairy2i_convert(GOOD, 0, 4, 4, GOOD, GOOD, 2, None) == 1
    assert lib.fairy2i_convert(GOOD, 4, 4, 3, GOOD, GOOD, 2, None) == 2       # ldR < cols
    assert lib.fairy2i_convert(GOOD, 4, 5, 5, GOOD, GOOD, 2, None) == 2       # ldc < m = 3
    assert lib.fairy2i_convert(GOOD, 4, 4, 4, ODD, GOOD, 2, None) == 3        # U not 8-aligned


def test_quantize_validation(lib):
    ws = lib.fairy2i_quantize_workspace_bytes(8, 8, 2)
    args = dict(U=GOOD, W=GOOD, n=8, m=8, ldc=8, T=2, codes=GOOD, scales=GOOD, ws=GOOD, wsb=ws)

    def call(**kw):
        a = dict(args, **kw)
        return lib.fairy2i_quantize(a["U"], a["W"], a["n"], a["m"], a["ldc"], a["T"], a["codes"],
                                    a["scales"], a["ws"], a["wsb"], None)
    assert call(T=0) == 1 and call(T=9) == 1 and call(U=None) == 1 and call(n=0) == 1
    assert call(ldc=7) == 2
    assert call(codes=ODD) == 3
    assert call(wsb=ws - 1) == 5 and call(ws=None) == 5
    assert call(ws=P((1 << 20) + 16)) == 3                                     # not 256-aligned


def test_wl_matmul_validation(lib):
    def call(x=GOOD, xdt=1, B=1, inf=16, ldx=16, codes=GOOD, scales=GOOD, outf=16, T=2, y=GOOD,
             ldy=16, path=0):
        return lib.fairy2i_wl_matmul_path(x, xdt, B, inf, ldx, codes, scales, outf, T, y, ldy,
                                          path, None)
    assert call(B=0) == 0                      # empty batch: nothing to do
    assert call(B=-1) == 1 and call(T=0) == 1 and call(path=6) == 1 and call(x=None) == 1
    assert call(path=2) == 1                   # retired
    assert call(path=5, T=5) == 1   # the chained kernel: T <= 4
    assert call(xdt=7) == 4
    assert call(ldx=15) == 2 and call(ldy=15) == 2
    assert call(x=ODD) == 3 and call(codes=ODD) == 3


def test_selftest_wait_timeout_validation(lib):
    """Out-of-range limits are refused before anything is enqueued."""
    assert lib.fairy2i_selftest_wait_timeout(0, None) == 1
    assert lib.fairy2i_selftest_wait_timeout(100001, None) == 1


def test_wl_matmul_group_validation(lib):
    arr = ctypes.c_void_p * 4

    def call(count=3, B=1, inf=16, ldx=16, outf=16, T=2, ldy=16, xdt=1, codes=None, ys=None,
             null_arrays=False):
        cp = arr(*([GOOD] * 4)) if codes is None else codes
        sp = arr(*([GOOD] * 4))
        yp = arr(*([GOOD] * 4)) if ys is None else ys
        if null_arrays:
            cp = sp = yp = None
        return lib.fairy2i_wl_matmul_group(GOOD, xdt, B, inf, ldx, count, cp, sp, outf, T, yp,
                                           ldy, None)
    assert call(B=0) == 0                                    # empty batch: nothing to do
    assert call(count=0) == 1 and call(count=5) == 1 and call(null_arrays=True) == 1
    assert call(T=0) == 1 and call(xdt=7) == 4
    assert call(ldx=15) == 2 and call(ldy=15) == 2
    assert call(codes=arr(GOOD, ODD, GOOD, GOOD)) == 3        # a misaligned member
    assert call(ys=arr(GOOD, GOOD, None, GOOD)) == 1          # a null member
    # the group call with an explicit kernel: only paths 0, 1, 3, 4 and 5 exist for a group
    cp = arr(*([GOOD] * 4))
    for path in (2, 6, -1):
        assert lib.fairy2i_wl_matmul_group_path(GOOD, 1, 1, 16, 16, 3, cp, cp, 16, 2, cp, 16,
                                                path, None) == 1
    # path 3 (the prefill GEMM) outside its domain, rejected before any launch: float32 x, and
    # m = 6 complex inputs (m % 8 != 0)
    assert lib.fairy2i_wl_matmul_group_path(GOOD, 0, 1, 16, 16, 3, cp, cp, 16, 2, cp, 16, 3,
                                            None) == 1
    assert lib.fairy2i_wl_matmul_group_path(GOOD, 1, 1, 12, 16, 3, cp, cp, 16, 2, cp, 16, 3,
                                            None) == 1
    assert lib.fairy2i_wl_matmul_group_path(GOOD, 1, 0, 16, 16, 3, cp, cp, 16, 2, cp, 16, 4,
                                            None) == 0     # empty batch on path 4


def test_codes_adjoint_validation(lib):
    assert lib.fairy2i_codes_adjoint(None, 4, 4, 2, GOOD, None) == 1
    assert lib.fairy2i_codes_adjoint(GOOD, 0, 4, 2, P((1 << 24)), None) == 1
    assert lib.fairy2i_codes_adjoint(GOOD, 4, 4, 9, P((1 << 24)), None) == 1
    assert lib.fairy2i_codes_adjoint(ODD, 4, 4, 2, P((1 << 24)), None) == 3
    assert lib.fairy2i_codes_adjoint(GOOD, 4, 4, 2, GOOD, None) == 1     # overlapping buffers


def test_wl_matmul_chain_validation(lib):
    """The chained decode refuses bad calls before anything is enqueued."""
    from paper_2512_02901_gb300.binding import ChainCall
    assert lib.fairy2i_wl_matmul_chain_max_calls() >= 128
    assert lib.fairy2i_wl_matmul_chain_workspace_bytes(1) == 0
    assert lib.fairy2i_wl_matmul_chain_workspace_bytes(128) >= 128 * 4

    def good():
        k = ChainCall()
        k.x, k.xdt, k.count, k.in_features, k.out_features = GOOD, 1, 1, 4096, 4096
        k.codes[0] = k.scales[0] = k.y[0] = GOOD
        return k

    def call(mod=None, n=1, T=2, cluster=0, ws=GOOD, wsb=1 << 20):
        arr = (ChainCall * n)(*[good() for _ in range(n)])
        if mod:
            mod(arr[n - 1])
        return lib.fairy2i_wl_matmul_chain(ctypes.cast(arr, ctypes.c_void_p), n, T, cluster, ws,
                                           wsb, None)

    assert call(T=0) == 1 and call(T=5) == 1 and call(cluster=3) == 1
    assert lib.fairy2i_wl_matmul_chain(None, 1, 2, 0, None, 0, None) == 1
    assert call(lambda k: setattr(k, "count", 0)) == 1
    assert call(lambda k: setattr(k, "count", 5)) == 1
    assert call(lambda k: setattr(k, "in_features", 24577)) == 1     # longer rows than the kernel takes
    assert call(lambda k: setattr(k, "x", None)) == 1
    assert call(lambda k: setattr(k, "xdt", 7)) == 4
    assert call(lambda k: setattr(k, "x", ODD)) == 3
    assert call(lambda k: k.codes.__setitem__(0, ODD)) == 3
    assert call(lambda k: k.y.__setitem__(0, None)) == 1
    assert call(n=3, ws=None, wsb=0) == 5                        # counters need a workspace
    assert call(n=3, wsb=8) == 5
    assert call(n=3, ws=ODD) == 3
