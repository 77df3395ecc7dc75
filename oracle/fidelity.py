"""Fidelity measures at the first generated-token step (test infrastructure).

* KL(p* || p) with p* = softmax(z*) of fresh recomputation and p = softmax(z)
  of the recovered cache (Section S2.1: forward KL, fresh as reference).
* top-1 agreement on the same distributions.
* Tail influence v_l = z^(l) - z^(l+1), T_b = sum_{l >= b} ||v_l||_2 (Eq. 2, Eq. S7)
  and the two certificates it gives: KL <= T_b^2 / 4 (Eq. 4) and top-1
  preservation when T_b < gamma*/2 (Eq. 5).
All in float64.
"""
from __future__ import annotations

from typing import Sequence

import numpy as np


def log_softmax(z: np.ndarray) -> np.ndarray:
    """log softmax of logits, row-wise (the next-token distributions p*, p of Section S2.1)."""
    z = np.asarray(z, dtype=np.float64)
    m = z.max(axis=-1, keepdims=True)
    return z - m - np.log(np.exp(z - m).sum(axis=-1, keepdims=True))


def kl(z_ref: np.ndarray, z: np.ndarray) -> np.ndarray:
    """sum_i p*_i (log p*_i - log p_i), row-wise, p* = softmax(z_ref), p = softmax(z): the forward
    KL with the fresh model as reference (Section S2.1)."""
    lr = log_softmax(z_ref)
    lc = log_softmax(z)
    return (np.exp(lr) * (lr - lc)).sum(axis=-1)


def top1_agree(z_ref: np.ndarray, z: np.ndarray) -> np.ndarray:
    """argmax agreement (ties resolve to the lowest index, as numpy does): top-1 agreement of
    Section S2.1."""
    return np.argmax(np.asarray(z_ref), axis=-1) == np.argmax(np.asarray(z), axis=-1)


def margin(z_ref: np.ndarray) -> np.ndarray:
    """gamma* = largest minus second-largest fresh logit: the margin of the top-1 certificate (Eq. 5,
    derived in Section S1.2)."""
    s = np.sort(np.asarray(z_ref, np.float64), axis=-1)
    return s[..., -1] - s[..., -2]


def tail_influence(z_hybrid: Sequence[np.ndarray]) -> np.ndarray:
    """T_b for b = 0..N from hybrid logits z^(0..N) (z^(N) = z*): T_b = sum_{l=b}^{N-1} ||z^(l) - z^(l+1)||
    (Eq. 2)."""
    z = [np.asarray(a, np.float64) for a in z_hybrid]
    n = len(z) - 1
    norms = np.array([np.linalg.norm(z[l] - z[l + 1]) for l in range(n)])
    return np.concatenate([np.cumsum(norms[::-1])[::-1], [0.0]])


def kl_certificate(t_b: float) -> float:
    """Upper bound T_b^2 / 4 on KL(p* || p^(b)) (Eq. 4)."""
    return 0.25 * t_b * t_b
