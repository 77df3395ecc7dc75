"""Versioned paged KV cache, fresh prefill, window restart and hybrid final logits.

Test infrastructure (see package docstring).

* The cache of a prefix under adapter version v_t is the per-layer set
  {K_l, V_l} (Eq. 1). It is stored here the way the GPU stores it: per layer a
  pool of 16-token pages [num_pages, Hkv, 16, d]; token t of a request lives at
  page ``page_table[t // 16]``, slot ``t % 16``.
* The executable restart (Section 4.2, "Executable restart") feeds the retained
  boundary state H_{r-1} (H_{-1} = the embedding, Section S1.1) through layers
  r..b-1 over the complete prefix under the current adapter and overwrites
  exactly those layers' K/V. Nothing else changes.
* The first-step next-token logits (Section 3.1; Section S2.1) of a recovered
  cache: the reading taken here is that the last prefix token is the first
  decode step. Its hidden state leaves the window at row n-1 and continues
  through layers e..N-1 as a single decode row whose attention reads that
  layer's cached K/V at positions < n-1 plus its own fresh k, v. For the window
  [0, N) this is exactly the last row of a fresh prefill (z^(N) = z*).
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Dict, List, Optional, Sequence

import numpy as np

from .decoder import (Dims, LayerAdapter, LayerParams, decode_row, decoder_layer, rmsnorm)

PAGE = 16


class PagedPool:
    """Per-layer K and V page pools, [num_pages, Hkv, 16, d] each: the layerwise cache of Eq. 1,
    stored in 16-token pages that requests address through page tables."""

    def __init__(self, n_layers: int, num_pages: int, n_kv_heads: int, head_dim: int,
                 dtype=np.float32):
        shape = (num_pages, n_kv_heads, PAGE, head_dim)
        self.k = [np.zeros(shape, dtype) for _ in range(n_layers)]
        self.v = [np.zeros(shape, dtype) for _ in range(n_layers)]

    @staticmethod
    def slots(page_table: np.ndarray, n: int):
        """(page, offset) of positions 0..n-1: page_table[t // 16], t % 16 (the Eq. 1 cache's layout)."""
        t = np.arange(n)
        return np.asarray(page_table)[t // PAGE], t % PAGE

    def write(self, layer: int, page_table: np.ndarray, k: np.ndarray, v: np.ndarray) -> None:
        """Store k/v [n, Hkv, d] of positions 0..n-1 of one request at its slots of ``layer``: the
        overwrite of a layer's K/V entries by recomputation (Section 4.2)."""
        pages, off = self.slots(page_table, k.shape[0])
        self.k[layer][pages, :, off, :] = k
        self.v[layer][pages, :, off, :] = v

    def read(self, layer: int, page_table: np.ndarray, n: int):
        """K, V [n, Hkv, d] of positions 0..n-1 of one request at ``layer`` (Eq. 1 entries)."""
        pages, off = self.slots(page_table, n)
        return self.k[layer][pages, :, off, :], self.v[layer][pages, :, off, :]

    def copy(self) -> "PagedPool":
        """An independent copy: a stale cache C^(t) kept while another is built (Eq. 1)."""
        out = PagedPool.__new__(PagedPool)
        out.k = [a.copy() for a in self.k]
        out.v = [a.copy() for a in self.v]
        return out


@dataclass
class Model:
    """Base model: per-layer params, embedding, final norm and LM head (float arrays); the frozen
    base of Section 2.1."""
    dims: Dims
    layers: List[LayerParams]
    embed: np.ndarray
    final_norm: np.ndarray
    lm_head: np.ndarray

    @property
    def n_layers(self) -> int:
        """N, the layers 0..N-1 of Eq. 1."""
        return len(self.layers)


@dataclass
class Adapter:
    """One adapter version theta_t: per-layer LoRA factors (Section 2.1, adapter evolution)."""
    layers: List[LayerAdapter]


@dataclass
class RequestCache:
    """Per-request state: tokens, page table and retained hidden states H_l (l = -1..N-1), the
    boundary states an executable restart reads (Section 4.2)."""
    tokens: np.ndarray
    page_table: np.ndarray
    hidden: Dict[int, np.ndarray] = field(default_factory=dict)

    @property
    def n(self) -> int:
        """n, the prefix length x_{1:n} of Eq. 1."""
        return int(self.tokens.shape[0])


def embed(model: Model, tokens: np.ndarray, dt=np.float32) -> np.ndarray:
    """H_{-1} = E[tokens] (Section S1.1)."""
    return np.asarray(model.embed[np.asarray(tokens)], dtype=dt)


def run_window(model: Model, adapter: Adapter, pool: PagedPool, req: RequestCache, s: int, e: int,
               dt=np.float32, chunk: int = 512, restart: Optional[np.ndarray] = None) -> np.ndarray:
    """Execute layers [s, e) over the complete prefix from the boundary state (Section 4.2).

    The boundary state is ``restart`` when given, else H_{s-1} from ``req.hidden`` (the
    embedding when s = 0). Overwrites the K/V of layers s..e-1 and sets H_l for those layers.
    Returns the last hidden state computed (H_{s-1} itself for an empty window).
    """
    if not (0 <= s <= e <= model.n_layers):
        raise ValueError("window out of range")
    if restart is not None:
        x = np.asarray(restart, dtype=dt)
    elif s == 0:
        x = embed(model, req.tokens, dt)
    else:
        x = np.asarray(req.hidden[s - 1], dtype=dt)
    for layer in range(s, e):
        x, k, v = decoder_layer(x, model.layers[layer], adapter.layers[layer], model.dims, dt, chunk)
        pool.write(layer, req.page_table, k, v)
        req.hidden[layer] = x
    return x


def prefill(model: Model, adapter: Adapter, pool: PagedPool, req: RequestCache, dt=np.float32,
            chunk: int = 512) -> np.ndarray:
    """Fresh full prefill: all N layers from the embedding; the cache C^(t) of Eq. 1."""
    req.hidden[-1] = embed(model, req.tokens, dt)
    return run_window(model, adapter, pool, req, 0, model.n_layers, dt, chunk)


def tail_decode(model: Model, adapter: Adapter, pool: PagedPool, req: RequestCache, e: int,
                h_row: np.ndarray, dt=np.float32) -> np.ndarray:
    """Carry row n-1 through layers e..N-1 against the cached K/V of those layers.

    Writes nothing: layers at and after the window end keep their historical cache. This is the
    hybrid execution of Section 3.1 with boundary b = e, the first-step state of Section S2.1.
    """
    n = req.n
    x = np.asarray(h_row, dtype=dt).reshape(1, -1)
    for layer in range(e, model.n_layers):
        kh, vh = pool.read(layer, req.page_table, n - 1)
        x, _, _ = decode_row(x, n - 1, kh, vh, model.layers[layer], adapter.layers[layer],
                             model.dims, dt)
    return x[0]


def logits(model: Model, h_final: np.ndarray, dt=np.float32) -> np.ndarray:
    """z = W_lm rmsnorm(h) * g_f for final hidden rows h [.., hidden]; returned in float64.

    The first-step next-token logits z of Section 3.1 (z* for the fresh row)."""
    hn = rmsnorm(np.atleast_2d(h_final), model.final_norm, model.dims.rms_eps, dt)
    return (hn @ np.asarray(model.lm_head, dtype=dt).T).astype(np.float64)


def recover(model: Model, adapter: Adapter, pool: PagedPool, req: RequestCache, s: int, e: int,
            dt=np.float32, chunk: int = 512, restart: Optional[np.ndarray] = None):
    """Bounded recovery R_{s, e-s} (Section S1.1) followed by the first-step final hidden row.

    Returns (H after the window [n, hidden], final hidden row after layer N-1 [hidden]).
    """
    x = run_window(model, adapter, pool, req, s, e, dt, chunk, restart)
    h_last = tail_decode(model, adapter, pool, req, e, x[-1], dt)
    return x, h_last
