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


def _bf16_proj(xin, P, A, m, bias):
    """One adapted projection as a bf16 tensor pipeline runs it (op outputs rounded to bf16)."""
    R = bf16_round
    y = xin @ P.W[m].T
    if bias and m in P.bias:
        y = y + P.bias[m]
    y = R(y)
    if m in A.AB:
        Am, Bm = A.AB[m]
        y = R(y + R(A.scale * R(R(xin @ Am.T) @ Bm.T)))
    return y


def bf16_layer_rows(x, P, A, dims, rows):
    """Layer output at `rows` (attention over all positions <= row) run as a bf16 tensor pipeline."""
    R = bf16_round
    n = x.shape[0]
    x = R(x)
    xn = R(Dec.rmsnorm(x, P.ln1, dims.rms_eps))
    cos, sin = Dec.rope_angles(np.arange(n), dims.head_dim, dims.rope_theta)
    q = R(Dec.apply_rope(_bf16_proj(xn, P, A, "q", True).reshape(n, dims.n_q_heads, dims.head_dim), cos, sin))
    k = R(Dec.apply_rope(_bf16_proj(xn, P, A, "k", True).reshape(n, dims.n_kv_heads, dims.head_dim), cos, sin))
    v = _bf16_proj(xn, P, A, "v", True).reshape(n, dims.n_kv_heads, dims.head_dim)
    out = []
    for t in rows:
        o = R(Dec.single_query_attention(q[t], k[:t + 1], v[:t + 1])).reshape(1, -1)
        x1 = R(x[t:t + 1] + _bf16_proj(o, P, A, "o", False))
        xn2 = R(Dec.rmsnorm(x1, P.ln2, dims.rms_eps))
        m = R(R(Dec.silu(_bf16_proj(xn2, P, A, "gate", False))) * _bf16_proj(xn2, P, A, "up", False))
        out.append(R(x1 + _bf16_proj(m, P, A, "down", False))[0])
    return np.stack(out)


def bf16_execution_recover(om, oa, pool, req, s, e, restart):
    """The window recovery executed the way a bf16 tensor pipeline runs it.

    The paper computes in bfloat16 throughout (Section 5.1): every op's output tensor is bf16
    while arithmetic inside an op accumulates in fp32. This runs the oracle's steps that way
    (projections, LoRA factors, RoPE outputs, attention output, residual sums, norms, the MLP
    activation and the cache K/V all rounded to bf16 as they are produced); the last row then
    continues through the tail in fp32, as the decode path does. Its distance from the plain fp32
    oracle measures how strongly the problem at hand amplifies bf16 rounding (large when deep-layer
    adapters dominate and attention is near one-hot). Returns (per-layer K, V, H dicts, final row).
    """
    R = bf16_round
    dims = om.dims
    n = req.n
    proj = _bf16_proj

    cos, sin = Dec.rope_angles(np.arange(n), dims.head_dim, dims.rope_theta)
    x = R(restart)
    ks, vs, hs = {}, {}, {}
    for l in range(s, e):
        P, A = om.layers[l], oa.layers[l]
        xn = R(Dec.rmsnorm(x, P.ln1, dims.rms_eps))
        q = proj(xn, P, A, "q", True).reshape(n, dims.n_q_heads, dims.head_dim)
        k = proj(xn, P, A, "k", True).reshape(n, dims.n_kv_heads, dims.head_dim)
        v = proj(xn, P, A, "v", True).reshape(n, dims.n_kv_heads, dims.head_dim)
        q, k = R(Dec.apply_rope(q, cos, sin)), R(Dec.apply_rope(k, cos, sin))
        o = R(Dec.causal_gqa_attention(q, k, v))
        x1 = R(x + proj(o.reshape(n, -1), P, A, "o", False))
        xn2 = R(Dec.rmsnorm(x1, P.ln2, dims.rms_eps))
        mlp = R(R(Dec.silu(proj(xn2, P, A, "gate", False))) * proj(xn2, P, A, "up", False))
        x = R(x1 + proj(mlp, P, A, "down", False))
        pool.write(l, req.page_table, k, v)
        ks[l], vs[l], hs[l] = k, v, x
    final = C.tail_decode(om, oa, pool, req, e, x[-1])
    return ks, vs, hs, final
