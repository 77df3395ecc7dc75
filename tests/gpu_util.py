"""Helpers shared by the GPU parity tests: oracle objects from the same seeded tensors."""
from __future__ import annotations

import numpy as np
import torch

import synth
from oracle import build as obuild, cache as C, decoder as Dec
from oracle.decoder import LayerAdapter

# Tolerances stated for the recomputation path (bf16 compute, fp32 accumulate):
REL_KVH = 1e-2       # per-layer relative Frobenius error of K/V pages and hidden states
KL_ABS = 1e-3        # absolute KL error
DRIFT_REL = 1e-4     # relative drift error
# Where a layer's own conditioning keeps every bf16-storage implementation above REL_KVH, the
# bar is this factor times the distance that the same layer moves when the oracle's steps store
# their intermediate tensors in bf16 at the points the path does (``bf16_storage_layer``): the
# two round at the same points and differ only in fp32 accumulation order, which decides a few
# roundings differently (measured ratio GPU / storage model on whole layers: 0.9-1.1).
STORAGE_FACTOR = 1.25


def to_np(t: torch.Tensor) -> np.ndarray:
    return t.detach().to("cpu", torch.float32).numpy()


def rel_frob(a, b) -> float:
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30))


def oracle_model(dm) -> C.Model:
    cfg = dm.cfg
    layers = [obuild.layer_params(cfg, l, tensors=w) if w is not None else None
              for l, w in enumerate(dm.layers)]
    return C.Model(obuild.dims_of(cfg), layers,
                   to_np(dm.embed) if dm.embed is not None else None,
                   to_np(dm.final_norm) if dm.final_norm is not None else None,
                   to_np(dm.lm_head) if dm.lm_head is not None else None)


def oracle_adapter(da) -> C.Adapter:
    return C.Adapter([LayerAdapter({m: (to_np(a), to_np(b)) for m, (a, b) in d.items()},
                                   Dec.lora_scale(da.lcfg.alpha, da.lcfg.rank)) if d is not None else None
                      for d in da.layers])


def oracle_pool(pool) -> C.PagedPool:
    p = C.PagedPool.__new__(C.PagedPool)
    p.k = [to_np(t) for t in pool.k_pages]
    p.v = [to_np(t) for t in pool.v_pages]
    return p


def snapshot(pool):
    return [t.clone() for t in pool.k_pages], [t.clone() for t in pool.v_pages]


def slots(page_table, n):
    pt = page_table.to("cpu").numpy()
    t = np.arange(n)
    return pt[t // synth.PAGE_SIZE], t % synth.PAGE_SIZE


def request_kv(pool_layer: torch.Tensor, page_table, n) -> np.ndarray:
    pages, off = slots(page_table, n)
    a = to_np(pool_layer)
    return a[pages, :, off, :]


def untouched_mask(num_pages, page_tables_and_lengths):
    """Boolean [num_pages, 16] of slots no request of the call owns."""
    m = np.ones((num_pages, synth.PAGE_SIZE), bool)
    for pt, n in page_tables_and_lengths:
        pages, off = slots(pt, n)
        m[pages, off] = False
    return m


def free_slots(t: torch.Tensor, free: np.ndarray) -> torch.Tensor:
    """Entries of a pool layer [P, Hkv, 16, d] at the (page, slot) pairs where ``free`` is True."""
    m = torch.from_numpy(free).to(t.device)
    return t.permute(0, 2, 1, 3)[m]


def bf16_round(a) -> np.ndarray:
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).bfloat16().float().numpy()


def _storage_proj(xin, P, A, m, bias):
    Am, Bm = A.AB.get(m, (None, None))
    return Dec.lora_linear(xin, P.W[m], Am, Bm, A.scale, P.bias.get(m) if bias else None)


def _storage_qkv(x, P, A, dims):
    """q, K, V of every position as the path stores them (bf16), from the bf16 normalised input."""
    R = bf16_round
    n = x.shape[0]
    d = dims.head_dim
    xn = R(Dec.rmsnorm(x, P.ln1, dims.rms_eps))
    cos, sin = Dec.rope_angles(np.arange(n), d, dims.rope_theta)
    q = R(Dec.apply_rope(_storage_proj(xn, P, A, "q", True).reshape(n, dims.n_q_heads, d), cos, sin))
    k = R(Dec.apply_rope(_storage_proj(xn, P, A, "k", True).reshape(n, dims.n_kv_heads, d), cos, sin))
    v = R(_storage_proj(xn, P, A, "v", True).reshape(n, dims.n_kv_heads, d))
    return q, k, v


def _storage_post(x, o, P, A, dims):
    """Output projection, residual, MLP and residual of rows whose attention output is o (bf16 stores)."""
    R = bf16_round
    o = R(o.reshape(x.shape[0], -1))
    x1 = R(x + _storage_proj(o, P, A, "o", False))
    xn2 = R(Dec.rmsnorm(x1, P.ln2, dims.rms_eps))
    m = R(Dec.silu(_storage_proj(xn2, P, A, "gate", False)) * _storage_proj(xn2, P, A, "up", False))
    return R(x1 + _storage_proj(m, P, A, "down", False))


def _storage_attention_rows(q, k, v, rows, grp):
    """Attention of query rows t over keys 0..t with the softmax weights rounded to bf16 before the
    P.V product and normalised by the sum of the unrounded weights (fp64)."""
    d = q.shape[-1]
    scale = np.float32(1.0 / np.sqrt(d))
    out = np.empty((len(rows), q.shape[1], d), np.float32)
    for j, t in enumerate(rows):
        for h in range(q.shape[1]):
            g = h // grp
            sc = (k[:t + 1, g] @ q[t, h]) * scale
            p = np.exp(sc - sc.max())
            out[j, h] = (bf16_round(p) @ v[:t + 1, g]) / np.float32(p.sum(dtype=np.float64))
    return out


def bf16_storage_rows(x, P, A, dims, rows):
    """``bf16_storage_layer`` evaluated at the given rows only (H at ``rows``; K and V of every
    position, which those rows attend to)."""
    x = np.asarray(x, np.float32)
    q, k, v = _storage_qkv(x, P, A, dims)
    o = _storage_attention_rows(q, k, v, rows, dims.n_q_heads // dims.n_kv_heads)
    return _storage_post(x[rows], o, P, A, dims), k, v


def bf16_storage_layer(x, P, A, dims, chunk: int = 512):
    """One decoder layer (the oracle's steps and arithmetic: fp32 products, fp32 softmax with fp64
    sums) with every tensor that the recomputation path keeps in memory between its kernels
    rounded to bf16 once: the normalised inputs, q and the cached K and V (after rotation), the
    softmax weights entering the P.V product (normalised by the sum of the unrounded weights),
    the attention output, the residual after attention, the MLP activation and the layer output.
    This is the declared precision of the path (bf16 storage, fp32 accumulation) applied to the
    oracle; its distance from the fp32 oracle is how far that precision alone moves a layer.
    Returns (H, K, V) like ``decoder.decoder_layer``."""
    x = np.asarray(x, np.float32)
    n = x.shape[0]
    q, k, v = _storage_qkv(x, P, A, dims)
    grp = dims.n_q_heads // dims.n_kv_heads
    scale = np.float32(1.0 / np.sqrt(dims.head_dim))
    o = np.empty_like(q)
    for h in range(dims.n_q_heads):
        g = h // grp
        for i0 in range(0, n, chunk):
            i1 = min(n, i0 + chunk)
            sc = (q[i0:i1, h] @ k[:i1, g].T) * scale
            sc[np.arange(i1)[None, :] > np.arange(i0, i1)[:, None]] = -np.inf
            p = np.exp(sc - sc.max(axis=-1, keepdims=True))
            den = p.sum(axis=-1, keepdims=True, dtype=np.float64).astype(np.float32)
            o[i0:i1, h] = (bf16_round(p) @ v[:i1, g]) / den
    return _storage_post(x, o, P, A, dims), k, v


def local_layer_report(x_in, P, A, dims, got_h, got_k, got_v, tag, plain: bool = False):
    """The GPU's layer outputs (H, and the request's K/V of that layer, every position) against the
    oracle's layer run on the GPU's own input for that layer (its bf16 restart state or previous
    window output), so each layer is judged on its own arithmetic. Returns
    [(name, err, bar, storage distance)]: the bar is REL_KVH, or, unless ``plain``, STORAGE_FACTOR
    times the bf16-storage model's distance on the same input when that is larger."""
    want_h, want_k, want_v = Dec.decoder_layer(x_in, P, A, dims)
    if plain:
        dist = {"h": 0.0, "k": 0.0, "v": 0.0}
    else:
        sh, sk, sv = bf16_storage_layer(x_in, P, A, dims)
        dist = {"h": rel_frob(sh, want_h), "k": rel_frob(sk, want_k), "v": rel_frob(sv, want_v)}
    out = []
    for name, got, want in (("h", got_h, want_h), ("k", got_k, want_k), ("v", got_v, want_v)):
        out.append((f"{name}{tag}", rel_frob(got, want), max(REL_KVH, STORAGE_FACTOR * dist[name]),
                    dist[name]))
    return out
