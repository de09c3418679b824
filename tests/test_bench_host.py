"""Host-side logic of bench.py (CPU): the kernel each decode call of the 7B stack runs (mirroring
the library's automatic choice), the committed per-call DRAM bytes against the calls'
algorithmic bytes, and the byte count the decode metric divides by."""
import pytest

import bench
from paper_2512_02901_gb300 import synth

SMS = 152   # GB300


def _calls(layers=1, grouped=True):
    shapes = {name: (rows, cols) for (_, _, name, rows, cols) in bench.layer_shapes(1)}
    groups = bench.GROUPS if grouped else tuple((nm,) for g in bench.GROUPS for nm in g)
    calls = []
    for _ in range(layers):
        for g in groups:
            rows, cols = shapes[g[0]]
            calls.append(dict(rows=rows, cols=cols,
                              members=[dict(name=nm, rows=shapes[nm][0], cols=shapes[nm][1])
                                       for nm in g]))
    return calls


def test_projection_shapes_are_llama2_7b():
    assert {n: (r, c) for (n, r, c) in synth.PROJECTIONS} == {
        "q": (4096, 4096), "k": (4096, 4096), "v": (4096, 4096), "o": (4096, 4096),
        "gate": (11008, 4096), "up": (11008, 4096), "down": (4096, 11008)}


def test_automatic_kernel_per_call():
    """The automatic decode path runs the persistent tcgen05 kernel (one-token form) for every
    call; path 1 is the warp-MMA kernel, path 5 the chained kernel."""
    for c in _calls():
        assert bench.decode_kernel(c, 0, SMS) == "stream"
        assert bench.decode_kernel(c, 1, SMS) == "fp8"
        assert bench.decode_kernel(c, 4, SMS) == "stream"
        assert bench.decode_kernel(c, 5, SMS) == "chain"


@pytest.mark.parametrize("path", [0, 1])
def test_traffic_table_matches_algorithmic_bytes(path):
    """Every committed capture is within 1.5 % of its call's algorithmic bytes (no re-reads; the
    4 MB o projection reads ~58 KB of per-CTA operands besides its codes)."""
    for c in _calls():
        name = ",".join(m["name"] for m in c["members"])
        kern = bench.decode_kernel(c, path, SMS)
        algo = bench.call_bytes(c, 1)
        got = bench.DECODE_DRAM_BYTES[kern].get(name)
        if got is None:
            continue
        assert abs(got - algo) <= 0.015 * algo, (kern, name, got, algo)


def test_step_traffic_sums_the_calls():
    one = bench.decode_traffic(_calls(1), 1, 1, SMS)
    assert bench.decode_traffic(_calls(32), 1, 1, SMS) == pytest.approx(32 * one, rel=1e-12)
    assert bench.decode_traffic(_calls(1), 1, 2, SMS) is None


def test_decode_bytes_per_step():
    """Packed codes (2 bits per complex weight, T = 2) + scales + fp32 y of the 224 linears, and
    the bf16 x of the 128 calls (a grouped call reads its shared x once): the denominator of the
    decode GB/s."""
    total = sum(bench.call_bytes(c, 1) for c in _calls(32))
    assert total == 1_625_938_944
    codes = 32 * sum(2 * 2 * ((r + 1) // 2) * ((c + 1) // 2) // 4 for (_, r, c) in synth.PROJECTIONS)
    assert codes == 1_619_001_344   # T = 2 bits per real parameter of the 7B linears


def test_step_launches_follow_the_automatic_path():
    """One launch per grouped call on the automatic path at every batch the bench runs, the
    chained kernel's explicit path one per 4 tokens, T = 3 from 512 tokens two per call."""
    for B in (1, 2, 4, 5, 8, 16, 64, 2048):
        assert bench.step_launches(128, B, 0) == 128
    assert bench.step_launches(128, 8, 5) == 256
    assert bench.step_launches(128, 3, 5) == 128
    assert bench.step_launches(4, 512, 0, T=3) == 8
    assert bench.step_launches(4, 511, 0, T=3) == 4
