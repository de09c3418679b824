"""GPU parity of the decoder-layer calls against the CPU oracle: Hermitian attention over a key /
value cache (Eq. hermitian-score), RMS norm with a fused residual add, silu * up, and one
widely-linear decoder layer step end to end (every linear quantized, attention Hermitian).

Tolerances. Attention accumulates scores and value sums in two-float arithmetic, so its outputs
are within a few fp32 roundings: relative Frobenius <= 1e-5 and, per element,
|err| <= 1e-5 sum_l p_l |v_l| (the scale of that output). RMS norm and silu * up: relative
1e-6 per element. The decoder layer: relative Frobenius <= 1e-5 on the output and on each
intermediate (against the oracle evaluated on the inputs the GPU used)."""
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


def _cplx(t):
    a = np.asarray(t, np.float64)
    n = a.shape[-1] // 2
    return a[..., :n] + 1j * a[..., n:]


def _rel(got, want):
    got = np.asarray(got)
    got = got.astype(np.complex128) if np.iscomplexobj(got) else got.astype(np.float64)
    return np.linalg.norm(got - want) / np.linalg.norm(want)


@pytest.mark.parametrize("n,heads,L,amp", [
    (64, 1, 1, 1.0), (64, 2, 7, 1.0), (2048, 32, 1, 1.0), (2048, 32, 130, 1.0),
    (2048, 32, 4096, 1.0), (256, 4, 1000, 1.0), (96, 3, 33, 1.0), (256, 2, 50, 1.0),
    (300, 5, 17, 1.0), (2048, 32, 512, 6.0),   # large scores: a sharp softmax
])
def test_attention_matches_oracle(F, n, heads, L, amp):
    g = torch.Generator().manual_seed(n + 7 * L + heads)
    q = amp * torch.randn(2 * n, generator=g)
    K = amp * torch.randn(L, 2 * n, generator=g)
    V = torch.randn(L, 2 * n, generator=g)
    out = F.hermitian_attention(q.to(DEV), K.to(DEV), V.to(DEV), L, heads)
    assert F.get_status() == 0
    qo, Ko, Vo = _cplx(q.numpy()), _cplx(K.numpy()), _cplx(V.numpy())
    want = O.hermitian_attention(qo, Ko, Vo, heads)
    got = _cplx(out.cpu().numpy())
    assert _rel(got, want) <= 1e-5
    S = O.hermitian_scores(qo, Ko, heads)
    P = np.exp(S - S.max(axis=1, keepdims=True))
    P /= P.sum(axis=1, keepdims=True)
    dc = n // heads
    scale = np.einsum("hl,lhc->hc", P, np.abs(Vo).reshape(L, heads, dc)).reshape(n)
    assert np.all(np.abs(got - want) <= 1e-5 * scale + 1e-30)


def test_attention_reads_a_strided_cache_prefix(F):
    """Only the first L rows of caches with a longer row stride are read."""
    n, heads, L, Lmax = 128, 2, 9, 20
    g = torch.Generator().manual_seed(5)
    big = torch.randn(Lmax, 2 * n + 16, generator=g)
    Vbig = torch.randn(Lmax, 2 * n + 16, generator=g)
    big[L:] = float("nan")
    Vbig[L:] = float("nan")
    q = torch.randn(2 * n, generator=g)
    out = F.hermitian_attention(q.to(DEV), big.to(DEV)[:, : 2 * n], Vbig.to(DEV)[:, : 2 * n], L,
                                heads)
    assert F.get_status() == 0
    want = O.hermitian_attention(_cplx(q.numpy()), _cplx(big[:L, : 2 * n].numpy()),
                                 _cplx(Vbig[:L, : 2 * n].numpy()), heads)
    assert _rel(_cplx(out.cpu().numpy()), want) <= 1e-5


@pytest.mark.parametrize("B,d", [(1, 4096), (3, 1000), (2, 7)])
def test_rmsnorm_with_residual_and_silu(F, B, d):
    g = torch.Generator().manual_seed(B * d)
    h = torch.randn(B, d, generator=g)
    delta = torch.randn(B, d, generator=g)
    w = 1.0 + 0.1 * torch.randn(d, generator=g)
    hd, dd, wd = h.to(DEV), delta.to(DEV), w.to(DEV)
    out = F.rmsnorm(hd, wd, 1e-5, delta=dd, h_out=hd)            # in-place residual add
    assert F.get_status() == 0
    v = (h + delta).double().numpy()
    assert np.allclose(hd.cpu().numpy(), (h + delta).numpy(), rtol=0, atol=0)
    want = np.stack([O.rmsnorm(v[b], w.double().numpy(), 1e-5) for b in range(B)])
    assert np.max(np.abs(out.cpu().numpy() - want) / (np.abs(want) + 1e-30)) <= 1e-6
    out2 = F.rmsnorm(hd, wd, 1e-5, out=hd)                          # plain, in place
    want2 = np.stack([O.rmsnorm(v[b], w.double().numpy(), 1e-5) for b in range(B)])
    assert np.max(np.abs(out2.cpu().numpy() - want2) / (np.abs(want2) + 1e-30)) <= 1e-6
    gg, uu = torch.randn(B, d, generator=g) * 4, torch.randn(B, d, generator=g)
    m = F.silu_mul(gg.to(DEV), uu.to(DEV))
    assert F.get_status() == 0
    wantm = O.silu_mul(gg.double().numpy(), uu.double().numpy())
    assert np.max(np.abs(m.cpu().numpy() - wantm) / (np.abs(wantm) + 1e-30)) <= 1e-6


def _oracle_layer(F, layer, names):
    codes = {}
    for nm in names:
        c = layer.codes[nm]
        T = layer.T
        out_f, in_f = {"q": (layer.d, layer.d), "k": (layer.d, layer.d), "v": (layer.d, layer.d),
                       "o": (layer.d, layer.d), "gate": (layer.dff, layer.d),
                       "up": (layer.dff, layer.d), "down": (layer.d, layer.dff)}[nm]
        n, m = O.complex_dims(out_f, in_f)
        codes[nm] = (O.unpack_codes(c.cpu().numpy().view(np.uint32).reshape(-1), T, n, m),
                     layer.scales[nm].cpu().numpy())
    codes["w_attn"] = layer.w_attn.cpu().double().numpy()
    codes["w_mlp"] = layer.w_mlp.cpu().double().numpy()
    return codes


@pytest.mark.parametrize("d,dff,heads,steps,prefill", [(512, 1376, 4, 3, 0), (4096, 11008, 32, 1, 200)])
def test_decoder_layer_step_matches_oracle(F, d, dff, heads, steps, prefill):
    """Steps of one decoder layer on random weights, with a cache that already holds `prefill`
    random positions; every step's output against the oracle layer on the same state."""
    g = torch.Generator().manual_seed(d + steps)
    weights = {}
    for pi, (nm, out_f, in_f) in enumerate((("q", d, d), ("k", d, d), ("v", d, d), ("o", d, d),
                                            ("gate", dff, d), ("up", dff, d), ("down", d, dff))):
        weights[nm] = synth.student_t_weight(out_f, in_f, seed=7000 + 10 * d + pi).to(DEV)
    w_attn = (1.0 + 0.1 * torch.randn(d, generator=g)).to(DEV)
    w_mlp = (1.0 + 0.1 * torch.randn(d, generator=g)).to(DEV)
    layer = F.WLDecoderLayer(weights, w_attn, w_mlp, heads, max_len=prefill + steps)
    del weights
    ol = _oracle_layer(F, layer, F.WLDecoderLayer.NAMES)
    if prefill:
        layer.k_cache[:prefill] = torch.randn(prefill, d, generator=g).to(DEV)
        layer.v_cache[:prefill] = torch.randn(prefill, d, generator=g).to(DEV)
        layer.pos = prefill
    h = torch.randn(1, d, generator=g).to(DEV)
    delta = None
    for s in range(steps):
        h_in = (h + delta if delta is not None else h).cpu().double().numpy()[0]
        Kc = _cplx(layer.k_cache[: layer.pos].cpu().numpy())
        Vc = _cplx(layer.v_cache[: layer.pos].cpu().numpy())
        h1, dn = layer.step(h, delta)
        assert F.get_status() == 0
        want, k_new, v_new = O.decoder_layer(h_in, ol, Kc, Vc, heads, layer.eps)
        got = (h1 + dn).cpu().double().numpy()[0]
        assert _rel(got, want) <= 1e-5, f"step {s}: {_rel(got, want):.2e}"
        assert _rel(_cplx(layer.k_cache[layer.pos - 1].cpu().numpy()), k_new) <= 1e-5
        assert _rel(_cplx(layer.v_cache[layer.pos - 1].cpu().numpy()), v_new) <= 1e-5
        h, delta = h1.clone(), dn.clone()
