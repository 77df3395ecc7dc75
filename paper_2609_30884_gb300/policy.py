"""Host recovery policy over the device's drift outputs (Section 4.1-4.2, Eq. 6-9, Eq. S4).

The library computes per-(layer, module) adapter displacements on the GPU (``crf_drift``); this
module turns them into a recovery action: the restart layer r of an update (Eq. S4: the first
cache layer the update can change), per-layer risk q_l = s_l d_l (Eq. 8) against calibrated
sensitivities s_l (Eq. 7), the range end b_t = 1 + max{l : q_l >= 1} (Eq. 9) and the window
[r, b_t) -- or direct reuse -- and the anchor bookkeeping: only the refreshed layers move to the
current version (Section 4.2). Two ablations from Section 5 (RQ4) are policies of the same shape:
``drift_only`` applies one calibration-frozen drift threshold to every affected layer, and
``fixed`` refreshes the same h-layer window after every update.

Plain host arithmetic on Python floats; no device work happens here.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Iterable, List, Optional, Sequence, Tuple

MODULES = ("q", "k", "v", "o", "gate", "up", "down")
# An update of k or v at layer s changes layer s's own cache entries; q, o and the MLP only
# change what later layers see, so the first changed cache layer is s + 1 (Eq. S4).
_SAME_LAYER = frozenset(("k", "v"))
CANDIDATE_WINDOWS = (0, 1, 2, 4, 8, 16)


def first_changed_layer(module: str, layer: int, n_layers: int) -> int:
    """Earliest cache layer an update of ``module`` at ``layer`` can change (n_layers: none)."""
    if module not in MODULES and module != "mlp":
        raise ValueError(f"unknown module {module!r}")
    return layer if module in _SAME_LAYER else min(layer + 1, n_layers)


def restart_of(updates: Iterable[Tuple[str, int]], n_layers: int) -> Optional[int]:
    """Restart layer of a set of (module, layer) updates: the shallowest updated layer among
    those whose change reaches some cache layer; None when no cache layer is affected."""
    layers = [l for m, l in updates if first_changed_layer(m, l, n_layers) < n_layers]
    return min(layers) if layers else None


def window_candidates(r: int, n_layers: int, lengths: Sequence[int] = CANDIDATE_WINDOWS) -> List[int]:
    """Window lengths tried in offline calibration: each length clipped to the executable suffix,
    plus the whole suffix, ascending and without repeats."""
    suffix = n_layers - r
    return sorted(set(min(h, suffix) for h in lengths) | {suffix})


def calibrate_sensitivity(conditions: Sequence[Tuple[float, int, int]], n_layers: int,
                          tail: float = 0.05, floor: float = 1e-12) -> List[float]:
    """s_l from calibration conditions (d_i, r_i, h*_i) (Eq. 6-7).

    A condition labels layers r_i .. r_i + h*_i - 1 as needing recovery. For each layer the labelled
    drifts are sorted and the (floor(tail * count) + 1)-th smallest, floored, becomes delta_l;
    s_l = 1 / delta_l, and 0 for a layer no condition labels.
    """
    per_layer: List[List[float]] = [[] for _ in range(n_layers)]
    for d, r, h in conditions:
        for l in range(r, min(r + h, n_layers)):
            per_layer[l].append(d)
    s = []
    for ds in per_layer:
        if not ds:
            s.append(0.0)
            continue
        ds.sort()
        idx = int(math.floor(tail * len(ds)))  # 0-based index of the (floor(tail*n)+1)-th value
        s.append(1.0 / max(ds[idx], floor))
    return s


def layer_displacement(drift_sq: Sequence[Sequence[Sequence[float]]], weight_space: bool = True) -> List[float]:
    """Per-layer d_l from one ``crf_drift`` output [N][7][2] computed against each layer's own
    anchor: sqrt of the layer's summed squared weight-space (||dW||_F^2, index 0) or parameter-space
    (||dA||^2 + ||dB||^2, index 1) distances."""
    k = 0 if weight_space else 1
    return [math.sqrt(sum(max(0.0, float(row[k])) for row in layer)) for layer in drift_sq]


def state_displacement(drift_sq_vs_anchor: Sequence[Sequence[Sequence[float]]]) -> float:
    """||theta_t - theta_a||_2 over the whole adapter state, from one ``crf_drift`` output taken
    with version a as every layer's anchor (the literal reading of d_l in Eq. 8)."""
    return math.sqrt(sum(max(0.0, float(row[1])) for layer in drift_sq_vs_anchor for row in layer))


@dataclass
class RecoveryPolicy:
    """Chooses a window per update and tracks the per-layer anchor versions.

    mode: "risk" (Eq. 8-9 with per-layer sensitivities), "drift_only" (one threshold for every
    affected layer: q_l = d_l / threshold), "fixed" (always [r, r + fixed_len)), "suffix" (always
    [r, N), the exact affected suffix), "full" ([0, N)), "reuse" (never recompute).
    """
    n_layers: int
    mode: str = "risk"
    sensitivity: Sequence[float] = ()
    threshold: float = 0.0
    fixed_len: int = 2
    anchors: List[int] = field(default_factory=list)

    def __post_init__(self):
        if self.mode not in ("risk", "drift_only", "fixed", "suffix", "full", "reuse"):
            raise ValueError(f"unknown mode {self.mode!r}")
        if self.mode == "risk" and len(self.sensitivity) != self.n_layers:
            raise ValueError("risk mode needs one sensitivity per layer")
        if self.mode == "drift_only" and not self.threshold > 0:
            raise ValueError("drift_only mode needs a positive threshold")
        if not self.anchors:
            self.anchors = [0] * self.n_layers

    def risk(self, d: Sequence[float]) -> List[float]:
        if self.mode == "risk":
            return [s * x for s, x in zip(self.sensitivity, d)]
        if self.mode == "drift_only":
            return [x / self.threshold for x in d]
        raise ValueError(f"mode {self.mode!r} has no risk")

    def window(self, restart: Optional[int], d: Sequence[float] = ()) -> Tuple[int, int]:
        """[s, e) to recompute for an update with restart layer ``restart``; s == e is reuse."""
        n = self.n_layers
        if self.mode == "full":
            return (0, n)
        if restart is None or self.mode == "reuse":
            r = 0 if restart is None else restart
            return (r, r)
        r = restart
        if self.mode == "suffix":
            return (r, n)
        if self.mode == "fixed":
            return (r, min(n, r + self.fixed_len))
        q = self.risk(d)
        hit = [l for l in range(n) if q[l] >= 1.0]
        b = 1 + max(hit) if hit else None
        # only layers at or after the restart can need the new adapter's cache (Section 4.2)
        return (r, b) if b is not None and b > r else (r, r)

    def commit(self, window: Tuple[int, int], version: int) -> None:
        """The refreshed layers now hold caches of ``version``."""
        s, e = window
        for l in range(s, e):
            self.anchors[l] = version

    def fraction(self, window: Tuple[int, int]) -> float:
        return (window[1] - window[0]) / self.n_layers
