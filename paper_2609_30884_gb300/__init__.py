"""GB300-native bounded KV-cache recomputation (CacheReforge, arXiv 2609.30884).

Python binding of the C ABI in include/crf.h. Objects here hold the caller's
torch tensors and the ctypes structs that point into them; the calls marshal
pointers, sizes and the current CUDA stream into libcrf.so. Nothing in this
package computes any step of the path.

    ctx = Context(0)
    model = Model(dims, layers, embed, final_norm, lm_head)
    cur = Adapter(lora, layers)                      # {module: (A, B)} per layer
    pool = KVPool(k_pages, v_pages)                  # per-layer [P, Hkv, 16, d] bf16
    req = Request(page_table, s, e, tokens=..., hidden_in=..., hidden_out=[...],
                  final_hidden_out=...)
    ws = ctx.workspace(model, cur, [req])
    ctx.recompute_window(model, cur, pool, [req], ws)
    ctx.drift(model.dims_c, cur, anchors, out_sq, ctx.drift_workspace(...))
    ctx.kl(model, ref_hidden, cur_hidden, out_kl, ...)
"""
from __future__ import annotations

import ctypes
from ctypes import POINTER, byref, c_size_t, c_void_p
from typing import Dict, List, Optional, Sequence, Tuple

import torch

from . import abi
from .abi import CrfError

MODULES = ("q", "k", "v", "o", "gate", "up", "down")

__all__ = ["Context", "Model", "Adapter", "KVPool", "Request", "CrfError", "MODULES", "abi",
           "kl_logits_noalloc"]


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _stream(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


class Model:
    """Base model: dims plus per-layer weight tensors (bf16 on the device)."""

    def __init__(self, dims: dict, layers: Sequence[Dict[str, torch.Tensor]],
                 embed: Optional[torch.Tensor] = None, final_norm: Optional[torch.Tensor] = None,
                 lm_head: Optional[torch.Tensor] = None):
        self.tensors = (list(layers), embed, final_norm, lm_head)
        self.dims = dict(dims)
        self.dims_c = abi.ModelDims(dims["n_layers"], dims["hidden"], dims["n_q_heads"],
                                    dims["n_kv_heads"], dims["head_dim"], dims["ffn"],
                                    dims["vocab"], dims["rms_eps"], dims["rope_theta"],
                                    int(bool(dims["qkv_bias"])))
        n = dims["n_layers"]
        self._layers = (abi.LayerWeights * n)()
        for l, w in enumerate(layers):
            if w is None:
                continue
            lw = self._layers[l]
            for j, m in enumerate(MODULES):
                lw.W[j] = _ptr(w.get(f"W_{m}"))
            for j, m in enumerate(("q", "k", "v")):
                lw.bias[j] = _ptr(w.get(f"bias_{m}"))
            lw.ln1 = _ptr(w.get("ln1"))
            lw.ln2 = _ptr(w.get("ln2"))
        self.c = abi.Model(self.dims_c, self._layers, _ptr(embed), _ptr(final_norm), _ptr(lm_head))


class Adapter:
    """One adapter version: per-layer {module: (A [r, in], B [out, r])} bf16 device tensors."""

    def __init__(self, rank: int, alpha: float, modules: Sequence[str],
                 layers: Sequence[Optional[Dict[str, Tuple[torch.Tensor, torch.Tensor]]]]):
        self.layers = list(layers)
        mask = sum(1 << MODULES.index(m) for m in modules)
        n = len(layers)
        self._A = (c_void_p * (n * 7))()
        self._B = (c_void_p * (n * 7))()
        for l, d in enumerate(layers):
            if d is None:
                continue
            for m, (A, B) in d.items():
                j = MODULES.index(m)
                self._A[l * 7 + j] = A.data_ptr()
                self._B[l * 7 + j] = B.data_ptr()
        self.dims_c = abi.LoraDims(rank, alpha, mask)
        self.c = abi.Adapter(self.dims_c, self._A, self._B)


class KVPool:
    """Per-layer K and V page pools, bf16 [num_pages, Hkv, 16, d]."""

    def __init__(self, k_pages: Sequence[torch.Tensor], v_pages: Sequence[torch.Tensor]):
        self.k_pages, self.v_pages = list(k_pages), list(v_pages)
        n = len(self.k_pages)
        self._k = (c_void_p * n)(*[t.data_ptr() for t in self.k_pages])
        self._v = (c_void_p * n)(*[t.data_ptr() for t in self.v_pages])
        self.num_pages = int(self.k_pages[0].shape[0])
        self.c = abi.KVPool(self._k, self._v, self.num_pages)


class Request:
    """One cached prefix and the window [s, e) to refresh (see crf_request)."""

    def __init__(self, page_table: torch.Tensor, s: int, e: int, n_tokens: Optional[int] = None,
                 tokens: Optional[torch.Tensor] = None, hidden_in: Optional[torch.Tensor] = None,
                 hidden_out: Optional[Sequence[torch.Tensor]] = None,
                 final_hidden_out: Optional[torch.Tensor] = None):
        if n_tokens is None:
            n_tokens = int(tokens.shape[0]) if tokens is not None else int(hidden_in.shape[0])
        self.keep = (page_table, tokens, hidden_in, hidden_out, final_hidden_out)
        self._hout = None
        if hidden_out is not None:
            self._hout = (c_void_p * max(1, len(hidden_out)))(*[t.data_ptr() for t in hidden_out])
        self.c = abi.Request(n_tokens, s, e, page_table.data_ptr(), _ptr(tokens), _ptr(hidden_in),
                             self._hout, _ptr(final_hidden_out))


def _req_array(reqs: Sequence[Request]):
    arr = (abi.Request * len(reqs))()
    for i, r in enumerate(reqs):
        arr[i] = r.c
    return arr


class Context:
    """A library context on one CUDA device."""

    def __init__(self, device: int = 0):
        self.lib = abi.load()
        self.device = device
        h = c_void_p()
        abi.check(self.lib.crf_create(byref(h), device))
        self.h = h

    def close(self) -> None:
        if self.h:
            self.lib.crf_destroy(self.h)
            self.h = c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -------------------------------------------------------------- window
    def workspace_size(self, model: Model, adapter: Adapter, reqs: Sequence[Request]) -> int:
        n = c_size_t()
        arr = _req_array(reqs)
        abi.check(self.lib.crf_workspace_size(self.h, byref(model.c), byref(adapter.dims_c), arr,
                                              len(reqs), byref(n)))
        return n.value

    def workspace(self, model: Model, adapter: Adapter, reqs: Sequence[Request]) -> torch.Tensor:
        return torch.empty(max(256, self.workspace_size(model, adapter, reqs)), dtype=torch.uint8,
                           device=f"cuda:{self.device}")

    def recompute_window(self, model: Model, adapter: Adapter, pool: KVPool,
                         reqs: Sequence[Request], workspace: torch.Tensor, stream=None) -> None:
        arr = _req_array(reqs)
        abi.check(self.lib.crf_recompute_window(self.h, byref(model.c), byref(adapter.c),
                                                byref(pool.c), arr, len(reqs),
                                                workspace.data_ptr(), workspace.numel(),
                                                _stream(stream)))

    # -------------------------------------------------------------- generation
    @staticmethod
    def _decode_rows(positions: Sequence[int], page_tables: Sequence[torch.Tensor],
                     tokens: torch.Tensor):
        n = len(positions)
        arr = (abi.DecodeRow * n)()
        for i in range(n):
            arr[i] = abi.DecodeRow(int(positions[i]), page_tables[i].data_ptr(), tokens[i:i + 1].data_ptr())
        return arr

    def decode_workspace(self, model: Model, adapter: Adapter, positions: Sequence[int],
                         page_tables: Sequence[torch.Tensor], tokens: torch.Tensor) -> torch.Tensor:
        n = c_size_t()
        arr = self._decode_rows(positions, page_tables, tokens)
        abi.check(self.lib.crf_decode_workspace_size(self.h, byref(model.c), byref(adapter.dims_c), arr,
                                                     len(positions), byref(n)))
        return torch.empty(max(256, n.value), dtype=torch.uint8, device=f"cuda:{self.device}")

    def decode_step(self, model: Model, adapter: Adapter, pool: KVPool, positions: Sequence[int],
                    page_tables: Sequence[torch.Tensor], tokens: torch.Tensor, next_tokens: torch.Tensor,
                    workspace: torch.Tensor, logits: Optional[torch.Tensor] = None, stream=None) -> None:
        """One generated token per row: tokens[i] (device int32) sits at positions[i]; its K/V are
        written into the row's pages and next_tokens[i] receives the greedy next token."""
        arr = self._decode_rows(positions, page_tables, tokens)
        abi.check(self.lib.crf_decode_step(self.h, byref(model.c), byref(adapter.c), byref(pool.c), arr,
                                           len(positions), next_tokens.data_ptr(), _ptr(logits),
                                           workspace.data_ptr(), workspace.numel(), _stream(stream)))

    # -------------------------------------------------------------- drift
    def drift_workspace(self, dims_c, lora_dims_c) -> torch.Tensor:
        n = c_size_t()
        abi.check(self.lib.crf_drift_workspace_size(self.h, byref(dims_c), byref(lora_dims_c),
                                                    byref(n)))
        return torch.empty(max(256, n.value), dtype=torch.uint8, device=f"cuda:{self.device}")

    def drift(self, dims_c, cur: Adapter, anchors: Sequence[Adapter], out_sq: torch.Tensor,
              workspace: torch.Tensor, stream=None) -> None:
        arr = (POINTER(abi.Adapter) * len(anchors))(*[ctypes.pointer(a.c) for a in anchors])
        abi.check(self.lib.crf_drift(self.h, byref(dims_c), byref(cur.c), arr, out_sq.data_ptr(),
                                     workspace.data_ptr(), workspace.numel(), _stream(stream)))

    # -------------------------------------------------------------- KL
    def kl_workspace(self, n_rows: int, vocab: int, hidden: int = 0) -> torch.Tensor:
        n = c_size_t()
        abi.check(self.lib.crf_kl_workspace_size(self.h, n_rows, vocab, hidden, byref(n)))
        return torch.empty(max(256, n.value), dtype=torch.uint8, device=f"cuda:{self.device}")

    def kl(self, model: Optional[Model], ref: torch.Tensor, cur: torch.Tensor, out_kl: torch.Tensor,
           vocab: int, workspace: torch.Tensor, logits_out: Optional[torch.Tensor] = None,
           stream=None) -> None:
        abi.check(self.lib.crf_kl(self.h, byref(model.c) if model is not None else None,
                                  ref.data_ptr(), cur.data_ptr(), int(ref.shape[0]), vocab,
                                  out_kl.data_ptr(), _ptr(logits_out), workspace.data_ptr(),
                                  workspace.numel(), _stream(stream)))

    def check(self, stream=None) -> None:
        abi.check(self.lib.crf_check(self.h, _stream(stream)))

    def selftest_timeout(self, stream=None) -> None:
        """Launch the bounded-wait self-test (its wait runs out after 2 s); the next check()
        raises CRF_ETIMEOUT."""
        abi.check(self.lib.crf_selftest_timeout(self.h, _stream(stream)))

    # -------------------------------------------------------------- profiling
    def profile_enable(self, on: bool = True, max_launches: int = 8192) -> None:
        abi.check(self.lib.crf_profile_enable(self.h, int(on), max_launches))

    def profile_read(self) -> Dict[str, Tuple[float, int]]:
        """{kernel kind: (total device ms, launches)} since the last read; also '_dropped'."""
        k = 32
        names = ctypes.create_string_buffer(k * 32)
        ms = (ctypes.c_double * k)()
        cnt = (ctypes.c_int * k)()
        n = ctypes.c_int()
        dropped = ctypes.c_int()
        abi.check(self.lib.crf_profile_read(self.h, k, names, ms, cnt, byref(n), byref(dropped)))
        out = {}
        for i in range(n.value):
            name = names.raw[i * 32:(i + 1) * 32].split(b"\0", 1)[0].decode()
            out[name] = (ms[i], cnt[i])
        out["_dropped"] = (0.0, dropped.value)
        return out


def kl_logits_noalloc(device: int, z_ref: torch.Tensor, z_cur: torch.Tensor, out_kl: torch.Tensor,
                      stream=None) -> None:
    """crf_kl_logits_noalloc: KL(softmax(z_ref) || softmax(z_cur)) per row with no workspace.

    For callers that cannot allocate device memory at call time; the library's fixed device
    scratch serves every call, so calls must not overlap on the GPU. The tensors are checked
    here (fp32, contiguous, same shape, on ``device``, out_kl long enough) because the library
    receives only their addresses.
    """
    if z_ref.dim() != 2 or tuple(z_cur.shape) != tuple(z_ref.shape):
        raise ValueError("z_ref and z_cur must be 2-D [n_rows, vocab] of the same shape")
    for name, t in (("z_ref", z_ref), ("z_cur", z_cur), ("out_kl", out_kl)):
        if t.dtype != torch.float32 or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous float32 tensor")
        if t.device.type != "cuda" or t.device.index != device:
            raise ValueError(f"{name} must be on cuda:{device}")
    if out_kl.numel() < z_ref.shape[0]:
        raise ValueError("out_kl holds fewer entries than z_ref has rows")
    if stream is None:
        stream = torch.cuda.current_stream(device)
    lib = abi.load()
    abi.check(lib.crf_kl_logits_noalloc(device, z_ref.data_ptr(), z_cur.data_ptr(),
                                        int(z_ref.shape[0]), int(z_ref.shape[1]),
                                        out_kl.data_ptr(), _stream(stream)))
