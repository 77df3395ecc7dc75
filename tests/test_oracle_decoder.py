"""Pins of the oracle's decoder-layer arithmetic against library routines, closed forms and brute force."""
import itertools
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import decoder as D

RNG = np.random.default_rng(1234)


def _r(*shape, s=1.0):
    return RNG.standard_normal(shape) * s


def test_rmsnorm_matches_torch_rms_norm():
    x, g = _r(7, 96), 1 + 0.1 * _r(96)
    y = D.rmsnorm(x, g, 1e-6, np.float64)
    ref = F.rms_norm(torch.tensor(x), (96,), torch.tensor(g), 1e-6).numpy()
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-12)


def test_rmsnorm_closed_form_constant_row():
    # a row of constant c has rms |c|: the result is sign(c) * g (eps negligible)
    y = D.rmsnorm(np.full((1, 8), -3.0), np.arange(1, 9, dtype=float), 0.0, np.float64)
    np.testing.assert_allclose(y[0], -np.arange(1, 9), rtol=1e-15)


def test_silu_matches_torch():
    x = _r(1000, s=5)
    np.testing.assert_allclose(D.silu(x), F.silu(torch.tensor(x)).numpy(), rtol=1e-13, atol=1e-15)


def test_lora_unmerged_equals_merged():
    x, W, A, B = _r(5, 24), _r(40, 24), _r(4, 24), _r(40, 4)
    b = _r(40)
    y = D.lora_linear(x, W, A, B, 2.0, b, np.float64)
    ref = x @ D.merged_weight(W, A, B, 2.0).T + b
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-12)
    # no adapter: plain linear
    np.testing.assert_allclose(D.lora_linear(x, W, None, None, 2.0, None, np.float64), x @ W.T)


def test_rope_equals_complex_rotation():
    n, h, d, theta = 9, 3, 16, 1e4
    x = _r(n, h, d)
    pos = np.arange(n) * 37 + 5
    cos, sin = D.rope_angles(pos, d, theta)
    y = D.apply_rope(x, cos, sin, np.float64)
    half = d // 2
    inv = theta ** (-np.arange(half) * 2.0 / d)
    z = (x[..., :half] + 1j * x[..., half:]) * np.exp(1j * pos[:, None, None] * inv[None, None, :])
    np.testing.assert_allclose(y[..., :half], z.real, atol=1e-12)
    np.testing.assert_allclose(y[..., half:], z.imag, atol=1e-12)


def test_rope_relative_position_property():
    d = 32
    q, k = _r(1, 1, d), _r(1, 1, d)

    def dot(p1, p2):
        c1, s1 = D.rope_angles(np.array([p1]), d, 1e6)
        c2, s2 = D.rope_angles(np.array([p2]), d, 1e6)
        return float(np.sum(D.apply_rope(q, c1, s1, np.float64) * D.apply_rope(k, c2, s2, np.float64)))

    assert dot(10, 3) == pytest.approx(dot(107, 100), rel=1e-9)
    assert dot(0, 0) == pytest.approx(float(np.sum(q * k)), rel=1e-12)


def _brute_attention(q, k, v):
    n, hq, d = q.shape
    grp = hq // k.shape[1]
    out = np.zeros_like(q)
    for h, i in itertools.product(range(hq), range(n)):
        g = h // grp
        s = [sum(q[i, h, c] * k[j, g, c] for c in range(d)) / math.sqrt(d) for j in range(i + 1)]
        m = max(s)
        e = [math.exp(x - m) for x in s]
        z = sum(e)
        for c in range(d):
            out[i, h, c] = sum(e[j] * v[j, g, c] for j in range(i + 1)) / z
    return out


def test_attention_brute_force_tiny():
    q, k, v = _r(11, 4, 8), _r(11, 2, 8), _r(11, 2, 8)
    got = D.causal_gqa_attention(q, k, v, chunk=4, dt=np.float64)
    np.testing.assert_allclose(got, _brute_attention(q, k, v), rtol=1e-10, atol=1e-12)


def test_attention_matches_torch_sdpa_gqa():
    n, hq, hkv, d = 70, 6, 2, 16
    q, k, v = _r(n, hq, d), _r(n, hkv, d), _r(n, hkv, d)
    got = D.causal_gqa_attention(q, k, v, chunk=32, dt=np.float64)
    tq, tk, tv = (torch.tensor(t).transpose(0, 1)[None] for t in (q, k, v))
    ref = F.scaled_dot_product_attention(tq, tk, tv, is_causal=True, enable_gqa=True)[0]
    np.testing.assert_allclose(got, ref.transpose(0, 1).numpy(), rtol=1e-10, atol=1e-12)


@pytest.mark.parametrize("hq,hkv,d,n,chunk", [(28, 4, 128, 300, 128), (12, 2, 128, 257, 64), (4, 2, 64, 129, 512)],
                         ids=["7b-heads", "1.5b-heads", "tiny-heads"])
def test_attention_matches_torch_sdpa_at_model_head_shapes(hq, hkv, d, n, chunk):
    """The model families' head layouts (GQA 7:1 and 6:1 at d = 128, 2:1 at d = 64), lengths that
    leave a ragged last query chunk, fp64 against the library routine."""
    q, k, v = _r(n, hq, d), _r(n, hkv, d), _r(n, hkv, d)
    got = D.causal_gqa_attention(q, k, v, chunk=chunk, dt=np.float64)
    tq, tk, tv = (torch.tensor(t).transpose(0, 1)[None] for t in (q, k, v))
    ref = F.scaled_dot_product_attention(tq, tk, tv, is_causal=True, enable_gqa=True)[0]
    np.testing.assert_allclose(got, ref.transpose(0, 1).numpy(), rtol=1e-10, atol=1e-12)


def test_single_query_attention_is_last_row_of_causal():
    q, k, v = _r(13, 4, 8), _r(13, 2, 8), _r(13, 2, 8)
    full = D.causal_gqa_attention(q, k, v, dt=np.float64)
    row = D.single_query_attention(q[-1], k, v, np.float64)
    np.testing.assert_allclose(row, full[-1], rtol=1e-12, atol=1e-13)


def _tiny_layer(seed=0, bias=True, dims=None, wstd=0.2):
    rng = np.random.default_rng(seed)
    if dims is None:
        dims = D.Dims(hidden=32, n_q_heads=4, n_kv_heads=2, head_dim=8, ffn=48, rms_eps=1e-6,
                      rope_theta=1e4)
    h, qd, kvd, f = dims.hidden, dims.n_q_heads * dims.head_dim, dims.n_kv_heads * dims.head_dim, dims.ffn
    shapes = {"q": (qd, h), "k": (kvd, h), "v": (kvd, h), "o": (h, qd), "gate": (f, h),
              "up": (f, h), "down": (h, f)}
    W = {m: rng.standard_normal(s) * wstd for m, s in shapes.items()}
    b = {m: rng.standard_normal(shapes[m][0]) * 0.1 for m in ("q", "k", "v")} if bias else {}
    P = D.LayerParams(W, b, 1 + 0.1 * rng.standard_normal(h), 1 + 0.1 * rng.standard_normal(h))
    AB = {m: (rng.standard_normal((4, s[1])) * 0.1, rng.standard_normal((s[0], 4)) * 0.1)
          for m, s in shapes.items()}
    return dims, P, D.LayerAdapter(AB, 2.0)


def _torch_layer(x, dims, P, ad):
    """The same block composed from torch library ops in fp64, with merged adapter weights."""
    t = lambda a: torch.tensor(np.asarray(a, np.float64))
    Wm = {m: t(D.merged_weight(P.W[m], *ad.AB[m], ad.scale)) for m in P.W}
    n = x.shape[0]
    X = t(x)
    xn = F.rms_norm(X, (dims.hidden,), t(P.ln1), dims.rms_eps)
    q = F.linear(xn, Wm["q"], t(P.bias["q"])).view(n, dims.n_q_heads, dims.head_dim)
    k = F.linear(xn, Wm["k"], t(P.bias["k"])).view(n, dims.n_kv_heads, dims.head_dim)
    v = F.linear(xn, Wm["v"], t(P.bias["v"])).view(n, dims.n_kv_heads, dims.head_dim)
    half = dims.head_dim // 2
    inv = dims.rope_theta ** (-torch.arange(half, dtype=torch.float64) * 2 / dims.head_dim)
    rot = torch.polar(torch.ones(n, half, dtype=torch.float64),
                      torch.arange(n, dtype=torch.float64)[:, None] * inv[None])

    def rope(a):
        c = torch.complex(a[..., :half], a[..., half:]) * rot[:, None, :]
        return torch.cat([c.real, c.imag], -1)

    q, k = rope(q), rope(k)
    o = F.scaled_dot_product_attention(q.transpose(0, 1)[None], k.transpose(0, 1)[None],
                                       v.transpose(0, 1)[None], is_causal=True, enable_gqa=True)
    o = o[0].transpose(0, 1).reshape(n, -1)
    x1 = X + F.linear(o, Wm["o"])
    xn2 = F.rms_norm(x1, (dims.hidden,), t(P.ln2), dims.rms_eps)
    m = F.silu(F.linear(xn2, Wm["gate"])) * F.linear(xn2, Wm["up"])
    return (x1 + F.linear(m, Wm["down"])).numpy(), k.numpy(), v.numpy()


def test_decoder_layer_matches_library_composition():
    dims, P, ad = _tiny_layer()
    x = _r(19, 32)
    h, k, v = D.decoder_layer(x, P, ad, dims, np.float64, chunk=8)
    rh, rk, rv = _torch_layer(x, dims, P, ad)
    np.testing.assert_allclose(h, rh, rtol=1e-10, atol=1e-11)
    np.testing.assert_allclose(k, rk, rtol=1e-10, atol=1e-11)
    np.testing.assert_allclose(v, rv, rtol=1e-10, atol=1e-11)


def test_decoder_layer_matches_library_composition_at_head_dim_128():
    """Head dim 128 with GQA 7:1 and theta 1e6 (the model families' RoPE frequencies), a ragged
    last query chunk."""
    dims = D.Dims(hidden=256, n_q_heads=7, n_kv_heads=1, head_dim=128, ffn=320, rms_eps=1e-6,
                  rope_theta=1e6)
    dims, P, ad = _tiny_layer(4, dims=dims, wstd=0.06)
    x = _r(37, 256)
    h, k, v = D.decoder_layer(x, P, ad, dims, np.float64, chunk=16)
    rh, rk, rv = _torch_layer(x, dims, P, ad)
    np.testing.assert_allclose(h, rh, rtol=1e-9, atol=1e-10)
    np.testing.assert_allclose(k, rk, rtol=1e-9, atol=1e-10)
    np.testing.assert_allclose(v, rv, rtol=1e-9, atol=1e-10)


def test_decode_row_matches_prefill_last_row():
    dims, P, ad = _tiny_layer(3)
    x = _r(12, 32)
    h, k, v = D.decoder_layer(x, P, ad, dims, np.float64)
    hr, kr, vr = D.decode_row(x[-1], 11, k[:-1], v[:-1], P, ad, dims, np.float64)
    np.testing.assert_allclose(hr[0], h[-1], rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(kr, k[-1], rtol=1e-12, atol=1e-13)


def test_float32_path_close_to_float64():
    dims, P, ad = _tiny_layer(5)
    x = _r(16, 32)
    h64, _, _ = D.decoder_layer(x, P, ad, dims, np.float64)
    h32, _, _ = D.decoder_layer(x, P, ad, dims, np.float32)
    assert np.linalg.norm(h32 - h64) / np.linalg.norm(h64) < 1e-5


def test_lora_scale_is_alpha_over_rank():
    """The adapter update enters as (alpha / r) B A: rank 8, alpha 16 -> 2; rank 16, alpha 32 -> 2."""
    assert D.lora_scale(16.0, 8) == 2.0 and D.lora_scale(32.0, 16) == 2.0 and D.lora_scale(8.0, 4) == 2.0
    # doubling the rank with the same factors padded by zeros halves the update at fixed alpha
    W, A, B = _r(6, 5), _r(2, 5), _r(6, 2)
    A2 = np.concatenate([A, np.zeros_like(A)]); B2 = np.concatenate([B, np.zeros_like(B)], 1)
    d1 = D.merged_weight(W, A, B, D.lora_scale(4.0, 2)) - W
    d2 = D.merged_weight(W, A2, B2, D.lora_scale(4.0, 4)) - W
    np.testing.assert_allclose(d2, d1 / 2, rtol=1e-12, atol=1e-14)
