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


def _moved(t, device):
    return t.to(device) if t is not None else None


class DeviceModel:
    """Base weights of ``layers`` (others None), embedding / final norm / LM head on ``device``.

    The values are drawn on ``gen`` (default: on ``device`` itself) and moved to ``device``; the
    generator gives the same bits on every device."""

    def __init__(self, cfg: synth.ModelCfg, device="cuda", layers: Optional[Sequence[int]] = None,
                 with_head: bool = True, seed: int = 0, gen=None):
        self.cfg = cfg
        g = device if gen is None else gen
        want = set(range(cfg.n_layers)) if layers is None else set(layers)
        self.layers: List[Optional[Dict[str, torch.Tensor]]] = [
            {k: v.to(device) for k, v in synth.layer_weights(cfg, l, seed, g).items()} if l in want else None
            for l in range(cfg.n_layers)]
        self.embed = _moved(synth.embedding(cfg, seed, g), device) if with_head else None
        self.final_norm = _moved(synth.final_norm(cfg, seed, g), device) if with_head else None
        self.lm_head = _moved(synth.lm_head(cfg, seed, g), device) if with_head else None
        self.crf = crf.Model(dims_dict(cfg), self.layers, self.embed, self.final_norm, self.lm_head)


class DeviceAdapter:
    """Adapter version ``version`` of the workload adapter on ``device`` (drawn on ``gen``)."""

    def __init__(self, cfg: synth.ModelCfg, lcfg: synth.LoraCfg, version: int, device="cuda",
                 layers: Optional[Sequence[int]] = None, seed: int = 0, override=None, gen=None):
        g = device if gen is None else gen
        want = set(range(cfg.n_layers)) if layers is None else set(layers)
        self.layers = [{m: (a.to(device), b.to(device))
                        for m, (a, b) in synth.adapter_version(cfg, lcfg, version, l, seed, g).items()}
                       if l in want else None
                       for l in range(cfg.n_layers)]
        if override:
            for (l, m), ab in override.items():
                self.layers[l][m] = ab
        self.lcfg = lcfg
        self.crf = crf.Adapter(lcfg.rank, lcfg.alpha, lcfg.modules, self.layers)


def make_pool(cfg: synth.ModelCfg, num_pages: int, device="cuda", fill: Optional[str] = "zeros",
              seed: int = 0, std: float = 1.0, gen=None):
    """Per-layer K/V page pools; ``fill="random"`` draws synthetic historical K/V values (on ``gen``)."""
    shape = (num_pages, cfg.n_kv_heads, synth.PAGE_SIZE, cfg.head_dim)
    g = device if gen is None else gen
    ks, vs = [], []
    for l in range(cfg.n_layers):
        if fill == "random":
            ks.append(synth.bf16_normal(shape, "pool_k", l, std, seed, g).to(device))
            vs.append(synth.bf16_normal(shape, "pool_v", l, std, seed, g).to(device))
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


class Versions:
    """Adapter versions 0..T of one synthetic continual trajectory: version 0 is the workload
    adapter's version ``base_version``; version t adds t seeded N(0, std^2) steps to every entry of
    A and B of ``module`` at ``layer`` (``synth.trajectory_factors``), so versions differ only there."""

    def __init__(self, cfg, lcfg, layer: int, module: str, std: float, seed: int, device,
                 base_version: int = 1):
        self.cfg, self.lcfg, self.layer, self.module, self.std, self.seed = cfg, lcfg, layer, module, std, seed
        self.device, self.base_version = device, base_version
        self.base = DeviceAdapter(cfg, lcfg, base_version, device)
        self._layers: Dict[int, list] = {}
        self._ad: Dict[int, crf.Adapter] = {}

    def adapter(self, t: int) -> crf.Adapter:
        if t not in self._ad:
            layers = list(self.base.layers)
            if t > 0:
                d = dict(layers[self.layer])
                d[self.module] = synth.trajectory_factors(self.cfg, self.lcfg, self.base_version, self.layer,
                                                          self.module, t, self.std, self.seed, self.device)
                layers[self.layer] = d
            self._layers[t] = layers  # keeps the tensors alive for the pointers below
            self._ad[t] = crf.Adapter(self.lcfg.rank, self.lcfg.alpha, self.lcfg.modules, layers)
        return self._ad[t]
