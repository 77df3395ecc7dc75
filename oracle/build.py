"""Turn seeded synthetic tensors (``synth``) into oracle objects (test infrastructure).

Values are the bf16 numbers the GPU receives, upcast to float32 here. When a
``source`` dict of already-generated torch tensors is given (for example tensors
the generator produced on a GPU and copied to the host), those are used instead
of regenerating; they are the same bits either way.
"""
from __future__ import annotations

from typing import Dict, Iterable, List, Optional

import numpy as np
import torch

import synth
from .cache import Adapter, Model
from .decoder import Dims, LayerAdapter, LayerParams, lora_scale


def _np(t: torch.Tensor) -> np.ndarray:
    return t.detach().to("cpu", torch.float32).numpy()


def dims_of(cfg: synth.ModelCfg) -> Dims:
    """Input construction (no passage of the paper): the oracle's shape record of a model config."""
    return Dims(cfg.hidden, cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim, cfg.ffn, cfg.rms_eps,
                cfg.rope_theta)


def layer_params(cfg: synth.ModelCfg, layer: int, seed: int = 0,
                 tensors: Optional[Dict[str, torch.Tensor]] = None) -> LayerParams:
    """Input construction: one layer's base weights as the oracle's float arrays."""
    w = tensors if tensors is not None else synth.layer_weights(cfg, layer, seed)
    W = {m: _np(w[f"W_{m}"]) for m in synth.MODULES}
    bias = {m: _np(w[f"bias_{m}"]) for m in ("q", "k", "v") if f"bias_{m}" in w}
    return LayerParams(W, bias, _np(w["ln1"]), _np(w["ln2"]))


def layer_adapter(cfg: synth.ModelCfg, lcfg: synth.LoraCfg, version: int, layer: int,
                  seed: int = 0, tensors=None) -> LayerAdapter:
    """Input construction: one layer of adapter version ``version``, scaled by alpha / r."""
    ab = tensors if tensors is not None else synth.adapter_version(cfg, lcfg, version, layer, seed)
    return LayerAdapter({m: (_np(a), _np(b)) for m, (a, b) in ab.items()}, lora_scale(lcfg.alpha, lcfg.rank))


def model(cfg: synth.ModelCfg, seed: int = 0, layers: Optional[Iterable[int]] = None,
          with_head: bool = True) -> Model:
    """Input construction: the whole model (or only ``layers``; the others are left as None)."""
    want = set(range(cfg.n_layers)) if layers is None else set(layers)
    lp: List[Optional[LayerParams]] = [layer_params(cfg, l, seed) if l in want else None
                                       for l in range(cfg.n_layers)]
    emb = _np(synth.embedding(cfg, seed)) if with_head else None
    fn = _np(synth.final_norm(cfg, seed)) if with_head else None
    lm = _np(synth.lm_head(cfg, seed)) if with_head else None
    return Model(dims_of(cfg), lp, emb, fn, lm)


def adapter(cfg: synth.ModelCfg, lcfg: synth.LoraCfg, version: int, seed: int = 0,
            layers: Optional[Iterable[int]] = None) -> Adapter:
    """Input construction: adapter version ``version`` over all (or the given) layers."""
    want = set(range(cfg.n_layers)) if layers is None else set(layers)
    return Adapter([layer_adapter(cfg, lcfg, version, l, seed) if l in want else None
                    for l in range(cfg.n_layers)])
