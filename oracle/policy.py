"""Host recovery policy, written from Section 4 and Section S1.1 (test infrastructure).

* Invalidation onset r_KV(m, s) (Eq. S4): key/value updates at layer s can change
  layer s's cache; query, output and MLP updates first change layer s+1's cache
  (N is the "nothing invalidated" sentinel).
* Executable restart r(c) = s whenever some cache layer is affected (Section 4.1,
  range selection; Section S1.1 after Eq. S4).
* Candidate windows H_i = {min(h, N - r_i) : h in {0,1,2,4,8,16}} U {N - r_i}
  and the first safe window (Section 4.1, offline calibration).
* Labels y_{i,l} = 1[r_i <= l < r_i + h*_i] (Eq. 6).
* delta_l = max(d_{l,(floor(0.05 n_l) + 1)}, 1e-12) over the positive drifts,
  s_l = 1/delta_l (0 for no positives) (Eq. 7).
* q_l = s_l d_l, triggered when q_l >= 1 (Eq. 8); b_t = 1 + max triggered layer
  (Eq. 9); window [r, b_t) or direct reuse.
* Anchors of exactly the recomputed layers move to theta_t (Section 4.2).
* Normalised recomputation fraction (b_t - r) / N (Section 4.2).
"""
from __future__ import annotations

import math
from typing import Callable, Dict, List, Optional, Sequence, Tuple

KV_MODULES = ("k", "v")
NON_KV_MODULES = ("q", "o", "gate", "up", "down", "mlp")
CANDIDATE_H = (0, 1, 2, 4, 8, 16)


def r_kv(module: str, s: int, n_layers: int) -> int:
    """Earliest cache layer that can change after updating ``module`` at layer s (Eq. S4)."""
    if module in KV_MODULES:
        return s
    if module in NON_KV_MODULES:
        return min(s + 1, n_layers)
    raise ValueError(f"unknown module {module!r}")


def restart_layer(module: str, s: int, n_layers: int) -> Optional[int]:
    """r(c): restart at s if any cache layer is affected, else None (nothing to recover): the
    executable restart of Section 4.1 / Section 4.2 with the onset of Eq. S4."""
    return s if r_kv(module, s, n_layers) < n_layers else None


def candidate_windows(r: int, n_layers: int, hs: Sequence[int] = CANDIDATE_H) -> List[int]:
    """H_i: the distinct executable window lengths tried during calibration, ascending (the
    candidate set of the offline calibration, Section 4.1)."""
    return sorted({min(h, n_layers - r) for h in hs} | {n_layers - r})


def first_safe(cands: Sequence[int], safe: Callable[[int], bool]) -> Optional[int]:
    """h*_i = min{h in H_i : S_i(h) = 1} (first hit, no monotonicity assumed; Section 4.1)."""
    for h in sorted(cands):
        if safe(h):
            return h
    return None


def labels(r: int, h_star: int, n_layers: int) -> List[int]:
    """y_{i,l} = 1[r <= l < r + h*] for l = 0..N-1 (Eq. 6)."""
    return [1 if r <= l < r + h_star else 0 for l in range(n_layers)]


def sensitivity(drifts: Sequence[float], label_rows: Sequence[Sequence[int]], n_layers: int,
                tail: float = 0.05, floor: float = 1e-12) -> List[float]:
    """s_l from calibration conditions (Eq. 7).

    drifts[i] is d_i, label_rows[i][l] is y_{i,l}. For each layer, D+_l collects d_i with y = 1;
    delta_l is its (floor(tail * n_l) + 1)-th smallest value (1-based), floored at 1e-12.
    """
    out = []
    for l in range(n_layers):
        pos = sorted(d for d, y in zip(drifts, label_rows) if y[l])
        if not pos:
            out.append(0.0)
            continue
        k = math.floor(tail * len(pos)) + 1
        out.append(1.0 / max(pos[k - 1], floor))
    return out


def risk(sens: Sequence[float], disp: Sequence[float]) -> List[float]:
    """q_l(t) = s_l d_l(t) (Eq. 8)."""
    return [s * d for s, d in zip(sens, disp)]


def range_end(q: Sequence[float]) -> Optional[int]:
    """b_t = 1 + max{l : q_l >= 1}, or None when no layer is triggered (Eq. 9)."""
    trig = [l for l, v in enumerate(q) if v >= 1.0]
    return 1 + max(trig) if trig else None


def plan(r: Optional[int], q: Sequence[float]) -> Tuple[int, int]:
    """Recovery window [r, b_t); (r, r) (empty) means direct reuse.

    b_t <= r (only layers before the restart triggered) is read as reuse: layers before r
    are unaffected by the update (Section 4.2).
    """
    if r is None:
        return (0, 0)
    b = range_end(q)
    if b is None or b <= r:
        return (r, r)
    return (r, b)


def update_anchors(anchors: List[int], window: Tuple[int, int], version: int) -> List[int]:
    """theta_l^anchor <- theta_t for l in the refreshed window only (Section 4.2)."""
    s, e = window
    return [version if s <= l < e else a for l, a in enumerate(anchors)]


def recompute_fraction(window: Tuple[int, int], n_layers: int) -> float:
    """(b_t - r) / N (Section 4.2)."""
    return (window[1] - window[0]) / n_layers


def displacement(anchors: Sequence[int], version: int,
                 table_for: Callable[[int], Sequence[Sequence[float]]]) -> List[float]:
    """d_l(t) = ||theta_t - theta_l^anchor||_2 over the whole adapter state (Eq. 8, literal reading).

    ``table_for(a)`` returns the per-(layer, module) squared parameter distance between version
    ``version`` and anchor version ``a``; d_l sums it over every layer and module.
    """
    out = []
    for a in anchors:
        if a == version:
            out.append(0.0)
            continue
        t = table_for(a)
        out.append(math.sqrt(sum(sum(row) for row in t)))
    return out
