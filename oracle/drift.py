"""Adapter displacement between two versions, per layer and module (test infrastructure).

Eq. 8 writes the runtime displacement of layer l as d_l(t) = ||theta_t - theta_l^anchor||_2.
Two readings are produced per (layer, module), both as squared quantities so the
host can sum them over any set of modules or layers:

* parameter space:  ||A_1 - A_0||_F^2 + ||B_1 - B_0||_F^2
* weight space:     ||B_1 A_1 - B_0 A_0||_F^2  (the change of the unscaled LoRA
  update; multiply by (alpha/r)^2 for the effective weight change)

The weight-space value is computed densely (only on tiny shapes) and through the
rank-2r factorisation B_1 A_1 - B_0 A_0 = [B_1 - B_0 | B_0] [A_1 ; A_1 - A_0],
whose squared Frobenius norm is tr((Bt^T Bt)(At At^T)) with 2r x 2r Grams.
All in float64.
"""
from __future__ import annotations

import numpy as np


def param_sq(A0, B0, A1, B1) -> float:
    """||A_1 - A_0||_F^2 + ||B_1 - B_0||_F^2: one module's share of ||theta_t - theta^anchor||_2^2
    in Eq. 8 (the adapter compared as parameters)."""
    A0, B0, A1, B1 = (np.asarray(t, np.float64) for t in (A0, B0, A1, B1))
    return float(np.sum((A1 - A0) ** 2) + np.sum((B1 - B0) ** 2))


def dense_sq(A0, B0, A1, B1) -> float:
    """||B_1 A_1 - B_0 A_0||_F^2 formed explicitly: the weight-space reading of the Eq. 8
    displacement (tiny shapes only)."""
    A0, B0, A1, B1 = (np.asarray(t, np.float64) for t in (A0, B0, A1, B1))
    d = B1 @ A1 - B0 @ A0
    return float(np.sum(d * d))


def factored_sq(A0, B0, A1, B1) -> float:
    """The same weight-space displacement as ``dense_sq`` (Eq. 8) through the rank-2r factors and
    their 2r x 2r Grams."""
    A0, B0, A1, B1 = (np.asarray(t, np.float64) for t in (A0, B0, A1, B1))
    Bt = np.concatenate([B1 - B0, B0], axis=1)     # [out, 2r]
    At = np.concatenate([A1, A1 - A0], axis=0)     # [2r, in]
    gb = Bt.T @ Bt
    ga = At @ At.T
    return float(np.sum(gb * ga.T))


def drift_table(anchor_layers, cur_layers, modules, dense: bool = False) -> np.ndarray:
    """[N, 7, 2] table of (weight-space, parameter-space) squared drifts (Eq. 8, per layer against
    that layer's anchor, Section 4.2).

    ``anchor_layers[l]`` / ``cur_layers[l]`` map module -> (A, B). Modules without an adapter
    give zeros.
    """
    n = len(cur_layers)
    out = np.zeros((n, len(modules), 2), np.float64)
    for l in range(n):
        for j, m in enumerate(modules):
            if m not in cur_layers[l]:
                continue
            A0, B0 = anchor_layers[l][m]
            A1, B1 = cur_layers[l][m]
            out[l, j, 0] = (dense_sq if dense else factored_sq)(A0, B0, A1, B1)
            out[l, j, 1] = param_sq(A0, B0, A1, B1)
    return out
