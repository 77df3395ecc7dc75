"""Seeded synthetic inputs for the bounded-recomputation workloads.

This module is shared by the oracle-side tests, the GPU parity tests and the
benchmark. It holds none of the method's arithmetic: only

* the workload shapes (Qwen2.5-shaped decoders, LoRA rank and modules, prefix
  lengths, windows),
* a counter-based value generator (a murmur3 32-bit finalizer keyed by
  ``(seed, tensor name, layer)``), written with integer ``torch`` ops so the
  same bits come out on the CPU and on a GPU,
* recipes that turn those values into bf16 weights, adapter versions, token
  ids and page tables.

Every random number is a pure function of ``(seed, name, layer, element
index)``, so any single layer of a 28-layer model can be regenerated alone,
on whichever device needs it.

Normal variates use the Irwin-Hall sum of four 16-bit uniforms, centred and
scaled to unit variance: an integer sum turned into a float by one exact
conversion and one fp32 multiply, so the value is bit-identical on every
device. The tails are bounded at about 3.46 sigma; for random-init weights that
is immaterial.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace
from typing import Dict, List, Optional, Sequence, Tuple

import torch

__all__ = [
    "ModelCfg", "LoraCfg", "Workload", "MODULES", "PAGE_SIZE",
    "TINY", "QWEN15B", "QWEN7B", "LORA_TINY", "LORA_QWEN",
    "WORKLOADS", "workload", "module_shape",
    "uniform_u32", "normal", "bf16_normal", "layer_weights", "adapter_version",
    "embedding", "final_norm", "lm_head", "token_ids", "page_permutation",
    "batch_plan", "hidden_state",
]

PAGE_SIZE = 16
# Projection order used everywhere: attention q,k,v,o then MLP gate, up, down.
MODULES = ("q", "k", "v", "o", "gate", "up", "down")


@dataclass(frozen=True)
class ModelCfg:
    name: str
    n_layers: int
    hidden: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    vocab: int
    rms_eps: float
    rope_theta: float
    qkv_bias: bool


@dataclass(frozen=True)
class LoraCfg:
    rank: int
    alpha: float
    modules: Tuple[str, ...]
    a_std: float = 0.02
    b_std: float = 0.01
    # version k+1 = version k + N(0, (step_std * (1 + layer))^2) on A and B
    step_std: float = 0.005

    @property
    def mask(self) -> int:
        return sum(1 << MODULES.index(m) for m in self.modules)


@dataclass(frozen=True)
class Workload:
    """One seeded workload: model, adapter, prefix lengths and windows."""
    name: str
    model: ModelCfg
    lora: LoraCfg
    n_tokens: Tuple[int, ...]           # one prefix length per request
    windows: Tuple[Tuple[int, int], ...]  # [s, e) per request
    stale_gap: Tuple[int, ...]          # cache of request i built under v_{cur - gap_i}
    cur_version: int = 1
    seed: int = 0


TINY = ModelCfg("tiny", 4, 256, 4, 2, 64, 688, 1024, 1e-6, 1e4, False)
QWEN15B = ModelCfg("qwen2.5-1.5b-shape", 28, 1536, 12, 2, 128, 8960, 151936, 1e-6, 1e6, True)
QWEN7B = ModelCfg("qwen2.5-7b-shape", 28, 3584, 28, 4, 128, 18944, 152064, 1e-6, 1e6, True)
LORA_TINY = LoraCfg(8, 16.0, ("q", "k", "v", "o"))
LORA_QWEN = LoraCfg(16, 32.0, MODULES)


def module_shape(cfg: ModelCfg, m: str) -> Tuple[int, int]:
    """(out_features, in_features) of projection ``m``; weights are row-major [out, in]."""
    h, d = cfg.hidden, cfg.head_dim
    return {
        "q": (cfg.n_q_heads * d, h),
        "k": (cfg.n_kv_heads * d, h),
        "v": (cfg.n_kv_heads * d, h),
        "o": (h, cfg.n_q_heads * d),
        "gate": (cfg.ffn, h),
        "up": (cfg.ffn, h),
        "down": (h, cfg.ffn),
    }[m]


def batch_plan(model: ModelCfg, n_req: int, seed: int = 2,
               n_min: int = 2048, n_max: int = 16384, max_len: int = 4,
               max_gap: int = 4) -> Tuple[Tuple[int, ...], Tuple[Tuple[int, int], ...], Tuple[int, ...]]:
    """Per-request prefix length, window and stale gap for the batched workload.

    Lengths are uniform over [n_min, n_max], starts uniform over [0, N-1],
    window lengths uniform over 1..max_len clamped to N - s, gaps over 1..max_gap.
    """
    u = uniform_u32((n_req, 4), "batch_plan", 0, seed).tolist()
    ns, wins, gaps = [], [], []
    for a, b, c, g in u:
        n = n_min + a % (n_max - n_min + 1)
        s = b % model.n_layers
        ln = 1 + c % max_len
        e = min(s + ln, model.n_layers)
        ns.append(n)
        wins.append((s, e))
        gaps.append(1 + g % max_gap)
    return tuple(ns), tuple(wins), tuple(gaps)


def _workloads() -> Dict[str, Workload]:
    w = {}
    w["tiny"] = Workload("tiny: 4L h256 512 tokens window [2,4)", TINY, LORA_TINY,
                         (512,), ((2, 4),), (1,))
    w["1.5b-4k"] = Workload("1.5B-shape 4K prefix window [20,22)", QWEN15B, LORA_QWEN,
                            (4096,), ((20, 22),), (1,))
    w["1.5b-16k"] = Workload("1.5B-shape 16K prefix window [20,22)", QWEN15B, LORA_QWEN,
                             (16384,), ((20, 22),), (1,))
    for ln in (1, 2, 4):
        w[f"7b-16k-w{ln}"] = Workload(f"7B-shape 16K prefix window [14,{14 + ln})", QWEN7B,
                                      LORA_QWEN, (16384,), ((14, 14 + ln),), (1,))
    w["7b-16k-full"] = Workload("7B-shape 16K prefix full prefill [0,28)", QWEN7B, LORA_QWEN,
                                (16384,), ((0, 28),), (1,))
    ns, wins, gaps = batch_plan(QWEN7B, 8)
    w["7b-batch8"] = Workload("7B-shape batch of 8 prefixes 2K-16K, own windows, shared pool",
                              QWEN7B, LORA_QWEN, ns, wins, gaps, cur_version=4)
    return w


def workload(name: str) -> Workload:
    return WORKLOADS[name]


# ---------------------------------------------------------------------------
# Counter-based generator
# ---------------------------------------------------------------------------
_M32 = 0xFFFFFFFF


def _key32(seed: int, name: str, layer: int) -> int:
    """FNV-1a (32-bit) of ``"seed/name/layer"``."""
    h = 0x811C9DC5
    for ch in f"{seed}/{name}/{layer}".encode():
        h ^= ch
        h = (h * 0x01000193) & _M32
    return h


def _mul32(x: torch.Tensor, c: int) -> torch.Tensor:
    """(x * c) mod 2^32 for int64 tensors holding uint32 values, without int64 overflow."""
    lo = (x & 0xFFFF) * c
    hi = (((x >> 16) * c) & 0xFFFF) << 16
    return (lo + hi) & _M32


def _fmix32(x: torch.Tensor) -> torch.Tensor:
    """murmur3 32-bit finalizer."""
    x = x ^ (x >> 16)
    x = _mul32(x, 0x85EBCA6B)
    x = x ^ (x >> 13)
    x = _mul32(x, 0xC2B2AE35)
    x = x ^ (x >> 16)
    return x


def _hash(n: int, lane: int, key: int, device) -> torch.Tensor:
    """uint32 stream ``fmix(fmix(2*i + lane) ^ key)`` for i in [0, n), as int64."""
    if n >= (1 << 31):
        raise ValueError("tensor too large for the 32-bit counter")
    i = torch.arange(n, dtype=torch.int64, device=device)
    return _fmix32(_fmix32(i * 2 + lane) ^ key)


def uniform_u32(shape: Sequence[int], name: str, layer: int = 0, seed: int = 0,
                device="cpu") -> torch.Tensor:
    n = math.prod(shape)
    return _hash(n, 0, _key32(seed, name, layer), device).reshape(tuple(shape))


def normal(shape: Sequence[int], name: str, layer: int = 0, std: float = 1.0,
           seed: int = 0, device="cpu", mean: float = 0.0) -> torch.Tensor:
    """fp32 tensor ~ mean + std * IrwinHall4 (unit variance), bit-identical on any device."""
    n = math.prod(shape)
    key = _key32(seed, name, layer)
    a = _hash(n, 0, key, device)
    b = _hash(n, 1, key, device)
    s = (a & 0xFFFF) + (a >> 16) + (b & 0xFFFF) + (b >> 16)      # 0 .. 262140
    c = torch.tensor(std * math.sqrt(3.0) / 65536.0, dtype=torch.float32, device=device)
    z = (s - 131070).to(torch.float32) * c
    if mean != 0.0:
        z = z + torch.tensor(mean, dtype=torch.float32, device=device)
    return z.reshape(tuple(shape))


def bf16_normal(shape, name, layer=0, std=1.0, seed=0, device="cpu", mean=0.0) -> torch.Tensor:
    return normal(shape, name, layer, std, seed, device, mean).to(torch.bfloat16)


# ---------------------------------------------------------------------------
# Recipes
# ---------------------------------------------------------------------------
W_STD = 0.02
NORM_GAIN_STD = 0.1


def layer_weights(cfg: ModelCfg, layer: int, seed: int = 0, device="cpu") -> Dict[str, torch.Tensor]:
    """Base weights of one decoder layer, bf16.

    ``W_<m>`` row-major [out, in] ~ N(0, 0.02); ``bias_<q|k|v>`` ~ N(0, 0.02) when the
    model has qkv bias; RMSNorm gains ``ln1``/``ln2`` ~ 1 + N(0, 0.1^2) so a dropped
    gain is visible.
    """
    out = {}
    for m in MODULES:
        o, i = module_shape(cfg, m)
        out[f"W_{m}"] = bf16_normal((o, i), f"W_{m}", layer, W_STD, seed, device)
    if cfg.qkv_bias:
        for m in ("q", "k", "v"):
            out[f"bias_{m}"] = bf16_normal((module_shape(cfg, m)[0],), f"bias_{m}", layer,
                                           W_STD, seed, device)
    out["ln1"] = bf16_normal((cfg.hidden,), "ln1", layer, NORM_GAIN_STD, seed, device, 1.0)
    out["ln2"] = bf16_normal((cfg.hidden,), "ln2", layer, NORM_GAIN_STD, seed, device, 1.0)
    return out


def adapter_version(cfg: ModelCfg, lcfg: LoraCfg, version: int, layer: int, seed: int = 0,
                    device="cpu") -> Dict[str, Tuple[torch.Tensor, torch.Tensor]]:
    """LoRA factors of adapter version ``version`` at ``layer``: {m: (A [r,in], B [out,r])} bf16.

    Version 0: A ~ N(0, a_std^2), B ~ N(0, b_std^2), rounded to bf16. Version k adds k
    independent fp32 perturbations of std ``step_std * (1 + layer)`` to the fp32 value of
    version 0 (in order 1..k) and rounds once.
    """
    out = {}
    for m in lcfg.modules:
        o, i = module_shape(cfg, m)
        a = bf16_normal((lcfg.rank, i), f"A_{m}", layer, lcfg.a_std, seed, device).float()
        b = bf16_normal((o, lcfg.rank), f"B_{m}", layer, lcfg.b_std, seed, device).float()
        st = lcfg.step_std * (1 + layer)
        for k in range(1, version + 1):
            a = a + normal((lcfg.rank, i), f"dA_{m}_v{k}", layer, st, seed, device)
            b = b + normal((o, lcfg.rank), f"dB_{m}_v{k}", layer, st, seed, device)
        out[m] = (a.to(torch.bfloat16), b.to(torch.bfloat16))
    return out


def trajectory_factors(cfg: ModelCfg, lcfg: LoraCfg, base_version: int, layer: int, module: str,
                       t: int, std: float, seed: int = 0, device="cpu",
                       base_seed: int = 0) -> Tuple[torch.Tensor, torch.Tensor]:
    """(A, B) of ``module`` at ``layer`` after t updates of a continual trajectory: the factors of
    adapter version ``base_version`` (drawn with ``base_seed``), plus t independent fp32 steps
    ~ N(0, std^2) on every entry of A and of B (drawn with ``seed``, in order 1..t), rounded to
    bf16 once."""
    a, b = adapter_version(cfg, lcfg, base_version, layer, base_seed, device)[module]
    a, b = a.float(), b.float()
    for k in range(1, t + 1):
        a = a + normal(tuple(a.shape), f"traj_dA_{module}_{k}", layer, std, seed, device)
        b = b + normal(tuple(b.shape), f"traj_dB_{module}_{k}", layer, std, seed, device)
    return a.to(torch.bfloat16), b.to(torch.bfloat16)


def embedding(cfg: ModelCfg, seed: int = 0, device="cpu") -> torch.Tensor:
    return bf16_normal((cfg.vocab, cfg.hidden), "embed", 0, W_STD, seed, device)


def final_norm(cfg: ModelCfg, seed: int = 0, device="cpu") -> torch.Tensor:
    return bf16_normal((cfg.hidden,), "final_norm", 0, NORM_GAIN_STD, seed, device, 1.0)


def lm_head(cfg: ModelCfg, seed: int = 0, device="cpu") -> torch.Tensor:
    return bf16_normal((cfg.vocab, cfg.hidden), "lm_head", 0, W_STD, seed, device)


def token_ids(cfg: ModelCfg, n: int, request: int = 0, seed: int = 0, device="cpu") -> torch.Tensor:
    """int32 token ids uniform over [0, vocab)."""
    u = uniform_u32((n,), "tokens", request, seed, device)
    return (u % cfg.vocab).to(torch.int32)


def page_permutation(num_pages: int, seed: int = 1, device="cpu") -> torch.Tensor:
    """A random permutation of physical page ids 0..num_pages-1 (int32)."""
    u = uniform_u32((num_pages,), "pages", 0, seed, "cpu")
    key = u * (1 << 31) + torch.arange(num_pages, dtype=torch.int64)   # ties broken by index
    return torch.argsort(key).to(torch.int32).to(device)


def hidden_state(cfg: ModelCfg, n: int, name: str = "hidden", layer: int = 0, seed: int = 0,
                 device="cpu", std: float = 1.0) -> torch.Tensor:
    """A standalone bf16 hidden-state tensor [n, hidden] (used where no prefill precedes)."""
    return bf16_normal((n, cfg.hidden), name, layer, std, seed, device)


WORKLOADS = _workloads()
