"""Assemble seeded synthetic workloads into device tensors and library objects.

Shared by the GPU tests, ``__graft_entry__.smoke()`` and ``bench.py``. Values
come from ``synth`` (the counter-based generator); nothing here computes any
step of the recomputation path.
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional, Sequence

import torch

import synth
import paper_2609_30884_gb300 as crf


def dims_dict(cfg: synth.ModelCfg) -> dict:
    return dict(n_layers=cfg.n_layers, hidden=cfg.hidden, n_q_heads=cfg.n_q_heads,
                n_kv_heads=cfg.n_kv_heads, head_dim=cfg.head_dim, ffn=cfg.ffn, vocab=cfg.vocab,
                rms_eps=cfg.rms_eps, rope_theta=cfg.rope_theta, qkv_bias=cfg.qkv_bias)


class DeviceModel:
    """Base weights of ``layers`` (others None), embedding / final norm / LM head on ``device``."""

    def __init__(self, cfg: synth.ModelCfg, device="cuda", layers: Optional[Sequence[int]] = None,
                 with_head: bool = True, seed: int = 0):
        self.cfg = cfg
        want = set(range(cfg.n_layers)) if layers is None else set(layers)
        self.layers: List[Optional[Dict[str, torch.Tensor]]] = [
            synth.layer_weights(cfg, l, seed, device) if l in want else None
            for l in range(cfg.n_layers)]
        self.embed = synth.embedding(cfg, seed, device) if with_head else None
        self.final_norm = synth.final_norm(cfg, seed, device) if with_head else None
        self.lm_head = synth.lm_head(cfg, seed, device) if with_head else None
        self.crf = crf.Model(dims_dict(cfg), self.layers, self.embed, self.final_norm, self.lm_head)


class DeviceAdapter:
    def __init__(self, cfg: synth.ModelCfg, lcfg: synth.LoraCfg, version: int, device="cuda",
                 layers: Optional[Sequence[int]] = None, seed: int = 0, override=None):
        want = set(range(cfg.n_layers)) if layers is None else set(layers)
        self.layers = [synth.adapter_version(cfg, lcfg, version, l, seed, device) if l in want else None
                       for l in range(cfg.n_layers)]
        if override:
            for (l, m), ab in override.items():
                self.layers[l][m] = ab
        self.lcfg = lcfg
        self.crf = crf.Adapter(lcfg.rank, lcfg.alpha, lcfg.modules, self.layers)


def make_pool(cfg: synth.ModelCfg, num_pages: int, device="cuda", fill: Optional[str] = "zeros",
              seed: int = 0, std: float = 1.0):
    """Per-layer K/V page pools; ``fill="random"`` draws synthetic historical K/V values."""
    shape = (num_pages, cfg.n_kv_heads, synth.PAGE_SIZE, cfg.head_dim)
    ks, vs = [], []
    for l in range(cfg.n_layers):
        if fill == "random":
            ks.append(synth.bf16_normal(shape, "pool_k", l, std, seed, device))
            vs.append(synth.bf16_normal(shape, "pool_v", l, std, seed, device))
        else:
            ks.append(torch.zeros(shape, dtype=torch.bfloat16, device=device))
            vs.append(torch.zeros(shape, dtype=torch.bfloat16, device=device))
    return crf.KVPool(ks, vs)


def pages_needed(n_tokens: int) -> int:
    return (n_tokens + synth.PAGE_SIZE - 1) // synth.PAGE_SIZE


def split_page_tables(lengths: Sequence[int], num_pages: int, seed: int = 1, device="cuda"):
    """Disjoint page tables for requests of ``lengths`` drawn from one random permutation."""
    perm = synth.page_permutation(num_pages, seed)
    out, at = [], 0
    for n in lengths:
        k = pages_needed(n)
        out.append(perm[at:at + k].to(device))
        at += k
    if at > num_pages:
        raise ValueError("pool too small")
    return out
