"""Offline tail-influence sweep on the device kernels (Sections 3.1-3.2, Eq. 2-5).

For a stale cache and the current adapter, z^(b) are the first-step next-token logits when the
cache is refreshed below layer b and historical from layer b on: the last prefix row restarts from
the refreshed hidden state H_{b-1} and is carried through layers b..N-1 against the historical
pages (b = 0 restarts from the embedding; z^(N) = z* is the fresh model). The sweep runs the N+1
hybrid rows as empty-window ``crf_recompute_window`` calls, then one ``crf_kl`` call over all of
them with the fresh row as reference, and derives on the host:

* v_l = z^(l) - z^(l+1) and the tail influence T_b = sum_{l >= b} ||v_l||_2 (Eq. 2),
* the KL certificate KL(p* || p^(b)) <= T_b^2 / 4 (Eq. 4),
* the top-1 certificate T_b < gamma*/2 => argmax z^(b) = argmax z* (Eq. 5), gamma* the fresh
  margin between the two largest logits,
* the first boundary at or after the restart whose KL meets a tolerance (the recomputation
  horizon of Eq. 3 counted from the restart).
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import List, Optional, Sequence

import numpy as np
import torch

from . import Context, Model, Adapter, KVPool, Request


@dataclass
class TailSweep:
    logits: np.ndarray        # [N + 1, V] fp64: z^(0) .. z^(N)
    kl: np.ndarray            # [N + 1]: KL(p* || p^(b)) from the device reduction
    top1: np.ndarray          # [N + 1] bool: argmax z^(b) == argmax z*
    v_norm: np.ndarray        # [N]: ||v_l||_2
    tail: np.ndarray          # [N + 1]: T_b (T_N = 0)
    margin: float             # gamma*
    kl_certificate_holds: np.ndarray   # [N + 1] bool: KL <= T_b^2 / 4 (+ slack)
    top1_certificate_holds: np.ndarray  # [N + 1] bool: T_b >= gamma*/2 or top-1 kept

    def horizon(self, restart: int, tol: float) -> Optional[int]:
        """First window length h >= 0 (boundary restart + h) whose KL is within ``tol``."""
        for b in range(restart, len(self.kl)):
            if self.kl[b] <= tol:
                return b - restart
        return None


def hybrid_rows(ctx: Context, model: Model, adapter: Adapter, stale: KVPool, page_table: torch.Tensor,
                n_tokens: int, tokens: torch.Tensor, fresh_hidden: Sequence[torch.Tensor],
                out: torch.Tensor) -> None:
    """out[b] = the final hidden row of z^(b) for b = 0..N (bf16 [N + 1, hidden])."""
    N = len(fresh_hidden)
    ws = None
    for b in range(N + 1):
        if b == 0:
            req = Request(page_table, 0, 0, n_tokens=n_tokens, tokens=tokens, final_hidden_out=out[0])
        else:
            req = Request(page_table, b, b, n_tokens=n_tokens, hidden_in=fresh_hidden[b - 1],
                          final_hidden_out=out[b])
        if ws is None:
            ws = ctx.workspace(model, adapter, [req])
        ctx.recompute_window(model, adapter, stale, [req], ws)


def sweep(ctx: Context, model: Model, adapter: Adapter, stale: KVPool, page_table: torch.Tensor,
          n_tokens: int, tokens: torch.Tensor, fresh_hidden: Sequence[torch.Tensor], vocab: int,
          kl_slack: float = 1e-4) -> TailSweep:
    """Run the N + 1 hybrid passes and the certificates for one stale cache and adapter."""
    N = len(fresh_hidden)
    dev = fresh_hidden[0].device
    hidden = fresh_hidden[0].shape[1]
    rows = torch.empty(N + 1, hidden, dtype=torch.bfloat16, device=dev)
    hybrid_rows(ctx, model, adapter, stale, page_table, n_tokens, tokens, fresh_hidden, rows)
    ref = rows[N:N + 1].expand(N + 1, hidden).contiguous()   # z^(N) = z*: the fresh row
    out_kl = torch.empty(N + 1, dtype=torch.float32, device=dev)
    logits = torch.empty(2 * (N + 1), vocab, dtype=torch.float32, device=dev)
    ws = ctx.kl_workspace(N + 1, vocab, hidden)
    ctx.kl(model, ref, rows, out_kl, vocab, ws, logits_out=logits)
    ctx.check()
    return certificates(logits[N + 1:].double().cpu().numpy(), out_kl.double().cpu().numpy(), kl_slack)


def certificates(z: np.ndarray, kl: np.ndarray, kl_slack: float = 1e-4) -> TailSweep:
    """The host side of the sweep from the hybrid logits z [N + 1, V] (z[N] = z*) and their KLs."""
    z = np.asarray(z, np.float64)
    kl = np.asarray(kl, np.float64)
    z_star = z[-1]
    v_norm = np.linalg.norm(z[:-1] - z[1:], axis=1)
    tail = np.concatenate([np.cumsum(v_norm[::-1])[::-1], [0.0]])
    top = np.sort(z_star)
    margin = float(top[-1] - top[-2])
    top1 = np.argmax(z, axis=1) == np.argmax(z_star)
    return TailSweep(z, kl, top1, v_norm, tail, margin,
                     kl <= 0.25 * tail * tail + kl_slack,
                     (tail >= margin / 2) | top1)
