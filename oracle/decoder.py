"""One decoder layer, written plainly (test infrastructure; see package docstring).

The layer maps (H_{l-1}; theta_l) to (H_l, C_l) as in Eq. S1: the hidden state
after the layer and the cache (post-rotation K, V) it writes. The projections
are Eq. S3 with the bias and rotation that Eq. S3 suppresses restored, and every
projection W of module m is the base weight plus the unmerged rank-r adapter,
W + (alpha/r) B A, kept unmerged (Section 5.1, "rank-8 LoRA adapter").

Block structure (Qwen2.5, the model family of Section 5.1):
    xn  = rmsnorm(x) * g1
    q,k,v = lora_linear(xn, ...) ; q,k = rope(q), rope(k)
    o   = causal GQA softmax attention(q, k, v)
    x1  = x + lora_linear(o, W_o)
    xn2 = rmsnorm(x1) * g2
    m   = silu(lora_linear(xn2, W_gate)) * lora_linear(xn2, W_up)
    x2  = x1 + lora_linear(m, W_down)
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Dict, Optional, Tuple

import numpy as np

MODULES = ("q", "k", "v", "o", "gate", "up", "down")


@dataclass
class Dims:
    """Shape of the decoder block of the model family in Section 5.1 (Qwen2.5)."""
    hidden: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    rms_eps: float
    rope_theta: float


def rmsnorm(x: np.ndarray, g: np.ndarray, eps: float, dt=np.float32) -> np.ndarray:
    """Row-wise RMSNorm: x / sqrt(mean(x^2) + eps) * g, mean-square accumulated in fp64.

    The normalisation of the block input that Section S1.1 writes as the bar in H-bar (Eq. S3)."""
    x = np.asarray(x, dtype=dt)
    ms = np.mean(np.square(x.astype(np.float64)), axis=-1, keepdims=True)
    inv = (1.0 / np.sqrt(ms + eps)).astype(dt)
    return (x * inv) * np.asarray(g, dtype=dt)


def lora_linear(x: np.ndarray, W: np.ndarray, A: Optional[np.ndarray], B: Optional[np.ndarray],
                scale: float, bias: Optional[np.ndarray] = None, dt=np.float32) -> np.ndarray:
    """y = x W^T (+ b) + scale * (x A^T) B^T with W [out,in], A [r,in], B [out,r] (unmerged LoRA).

    A projection of Eq. S3 under the current adapter: frozen base weight plus the adapter's
    low-rank update (Section 2.1, Section 5.1)."""
    x = np.asarray(x, dtype=dt)
    y = x @ np.asarray(W, dtype=dt).T
    if bias is not None:
        y = y + np.asarray(bias, dtype=dt)
    if A is not None:
        xa = x @ np.asarray(A, dtype=dt).T
        y = y + dt(scale) * (xa @ np.asarray(B, dtype=dt).T)
    return y


def rope_angles(positions: np.ndarray, head_dim: int, theta: float) -> Tuple[np.ndarray, np.ndarray]:
    """cos/sin of p * theta^(-2i/d) for i < d/2, computed in fp64. Shapes [n, d/2].

    The positional rotation that Eq. S3 suppresses, in the model family's rotate-half form."""
    i = np.arange(head_dim // 2, dtype=np.float64)
    inv_freq = theta ** (-2.0 * i / head_dim)
    ang = np.asarray(positions, dtype=np.float64)[:, None] * inv_freq[None, :]
    return np.cos(ang), np.sin(ang)


def apply_rope(x: np.ndarray, cos: np.ndarray, sin: np.ndarray, dt=np.float32) -> np.ndarray:
    """Rotate-half rotary embedding on x [n, H, d]: pairs (i, i + d/2) rotate by the angle of i.

    Applied to q and k before K is cached (the rotation Eq. S3 suppresses)."""
    x = np.asarray(x, dtype=dt)
    half = x.shape[-1] // 2
    c = cos.astype(dt)[:, None, :]
    s = sin.astype(dt)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def silu(x: np.ndarray) -> np.ndarray:
    """x * sigmoid(x), the gate of the SwiGLU MLP of the model family's block (Section 5.1)."""
    with np.errstate(over="ignore"):
        return x / (1.0 + np.exp(-x))


def _softmax_rows(s: np.ndarray) -> np.ndarray:
    s = s - s.max(axis=-1, keepdims=True)
    p = np.exp(s)
    return p / p.sum(axis=-1, keepdims=True, dtype=np.float64).astype(p.dtype)


def causal_gqa_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, chunk: int = 512,
                         dt=np.float32) -> np.ndarray:
    """softmax(q k^T / sqrt(d) + causal mask) v per query head, over the whole prefix.

    q [n, Hq, d], k/v [n, Hkv, d]; query head h reads kv head h // (Hq/Hkv). Query i sees keys
    j <= i. Query rows are processed in chunks only to bound memory. The self-attention of the
    block whose K, V form the cache of Eq. 1 (Eq. S3).
    """
    n, hq, d = q.shape
    hkv = k.shape[1]
    grp = hq // hkv
    scale = dt(1.0 / np.sqrt(d))
    q = np.asarray(q, dtype=dt)
    k = np.asarray(k, dtype=dt)
    v = np.asarray(v, dtype=dt)
    out = np.empty((n, hq, d), dtype=dt)
    for h in range(hq):
        g = h // grp
        for i0 in range(0, n, chunk):
            i1 = min(n, i0 + chunk)
            s = (q[i0:i1, h] @ k[:i1, g].T) * scale
            future = np.arange(i1)[None, :] > np.arange(i0, i1)[:, None]
            s[future] = -np.inf
            out[i0:i1, h] = _softmax_rows(s) @ v[:i1, g]
    return out


def single_query_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, dt=np.float32) -> np.ndarray:
    """One query row q [Hq, d] over keys k/v [t, Hkv, d] (all visible).

    The attention of a decoding row over a cache (Section 3.1: the first generated step)."""
    hq, d = q.shape
    grp = hq // k.shape[1]
    scale = dt(1.0 / np.sqrt(d))
    out = np.empty((hq, d), dtype=dt)
    for h in range(hq):
        g = h // grp
        s = (np.asarray(k[:, g], dt) @ np.asarray(q[h], dt)) * scale
        out[h] = _softmax_rows(s[None, :])[0] @ np.asarray(v[:, g], dt)
    return out


@dataclass
class LayerParams:
    """Base weights of one layer (float arrays holding the bf16 values): the frozen base model
    of Section 2.1."""
    W: Dict[str, np.ndarray]             # m -> [out, in]
    bias: Dict[str, np.ndarray]          # q/k/v -> [out] (empty when the model has none)
    ln1: np.ndarray
    ln2: np.ndarray


@dataclass
class LayerAdapter:
    """LoRA factors of one layer: m -> (A [r, in], B [out, r]); modules absent are unadapted.

    The layer's part theta_l of an adapter version (Section 2.1). ``scale`` multiplies B A
    (``lora_scale``)."""
    AB: Dict[str, Tuple[np.ndarray, np.ndarray]]
    scale: float


def lora_scale(alpha: float, rank: int) -> float:
    """alpha / r: the factor of the low-rank update B A in the LoRA parameterisation the paper
    adopts (Section 1, citing LoRA). Section 5.1 gives the adapter's rank but not alpha, which the
    workload fixes."""
    return float(alpha) / float(rank)


def _proj(x, P: LayerParams, ad: LayerAdapter, m: str, dt):
    A, B = ad.AB.get(m, (None, None))
    return lora_linear(x, P.W[m], A, B, ad.scale, P.bias.get(m), dt)


def qkv(x: np.ndarray, P: LayerParams, ad: LayerAdapter, dims: Dims, positions: np.ndarray,
        dt=np.float32):
    """Normalised input and post-rotation q, k plus v for rows ``x`` at ``positions`` (Eq. S3)."""
    n = x.shape[0]
    d = dims.head_dim
    xn = rmsnorm(x, P.ln1, dims.rms_eps, dt)
    q = _proj(xn, P, ad, "q", dt).reshape(n, dims.n_q_heads, d)
    k = _proj(xn, P, ad, "k", dt).reshape(n, dims.n_kv_heads, d)
    v = _proj(xn, P, ad, "v", dt).reshape(n, dims.n_kv_heads, d)
    cos, sin = rope_angles(positions, d, dims.rope_theta)
    return apply_rope(q, cos, sin, dt), apply_rope(k, cos, sin, dt), v


def post_attention(x: np.ndarray, o: np.ndarray, P: LayerParams, ad: LayerAdapter, dims: Dims,
                   dt=np.float32) -> np.ndarray:
    """Output projection + residual, then the SwiGLU MLP + residual: the rest of F_l in Eq. S1."""
    n = x.shape[0]
    x1 = np.asarray(x, dt) + _proj(o.reshape(n, -1), P, ad, "o", dt)
    xn2 = rmsnorm(x1, P.ln2, dims.rms_eps, dt)
    m = silu(_proj(xn2, P, ad, "gate", dt)) * _proj(xn2, P, ad, "up", dt)
    return x1 + _proj(m, P, ad, "down", dt)


def decoder_layer(x: np.ndarray, P: LayerParams, ad: LayerAdapter, dims: Dims,
                  dt=np.float32, chunk: int = 512):
    """(H_l, K_l, V_l) = (F_l, G_l)(H_{l-1}; theta_l) over a whole prefix at positions 0..n-1 (Eq. S1)."""
    n = x.shape[0]
    q, k, v = qkv(x, P, ad, dims, np.arange(n), dt)
    o = causal_gqa_attention(q, k, v, chunk, dt)
    return post_attention(x, o, P, ad, dims, dt), k, v


def decode_row(x_row: np.ndarray, pos: int, k_hist: np.ndarray, v_hist: np.ndarray,
               P: LayerParams, ad: LayerAdapter, dims: Dims, dt=np.float32):
    """One row at position ``pos`` attending to cached k/v at positions < pos plus its own fresh k, v.

    k_hist/v_hist [pos, Hkv, d] are the cached (historical) post-rotation keys and values of this
    layer. Returns (h_out [1, hidden], k_row, v_row). The row of a hybrid execution that reads
    historical states at this layer (Section 3.1).
    """
    q, k, v = qkv(x_row.reshape(1, -1), P, ad, dims, np.array([pos]), dt)
    kk = np.concatenate([np.asarray(k_hist, dt), k], axis=0)
    vv = np.concatenate([np.asarray(v_hist, dt), v], axis=0)
    o = single_query_attention(q[0], kk, vv, dt)
    return post_attention(x_row.reshape(1, -1), o[None], P, ad, dims, dt), k[0], v[0]


def merged_weight(W: np.ndarray, A: np.ndarray, B: np.ndarray, scale: float) -> np.ndarray:
    """W + scale * B A: the merged form of an adapted projection (used by the pins only); the same
    projection as ``lora_linear`` (Section 2.1)."""
    return np.asarray(W, np.float64) + scale * (np.asarray(B, np.float64) @ np.asarray(A, np.float64))
