"""Helpers shared by the GPU parity tests: oracle objects from the same seeded tensors."""
from __future__ import annotations

import numpy as np
import torch

import synth
from oracle import build as obuild, cache as C
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
                                   da.lcfg.scale) if d is not None else None
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
