"""A synthetic continual-adapter trajectory that drives the host recovery policy on the GPU kernels.

Section 5 (RQ4) replays 32 consecutive updates of one middle value projection and compares fresh
full prefill, the exact affected suffix, stale reuse, the drift-sensitive policy and two ablations
(one drift threshold for every layer; a fixed two-layer window), reporting per-version KL and top-1
agreement of the first-step distribution against the fresh model, the recomputed fraction, and
cache-maintenance time summed over the trajectory (Table 1, Table 2, Section S2). Here the inputs
are seeded and synthetic (random-init decoder of a Qwen2.5 shape, uniform token ids), the update is
one (layer, module) pair of the adapter moving by an N(0, std^2) step on every entry of A and B per
version, and the sensitivities come from a disjoint calibration trajectory (Eq. 6-7) with the
paper's acceptance rule for a candidate window (KL <= 0.05 and the top-1 token kept).

Maintenance = what a serving system runs per update: the drift queries the policy needs
(``crf_drift``), the window's ``crf_recompute_window`` (refreshing K/V pages and checkpoints), and
the host decision. The fresh reference and the evaluation of each method's first-step state are
measured outside it. Used by ``bench.py --case trajectory`` and the GPU tests, which supply the
synthetic adapter versions, token ids and page table.
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional, Sequence, Tuple

import torch

import paper_2609_30884_gb300 as crf
from paper_2609_30884_gb300 import policy as P

KL_SAFE = 0.05
METHODS = ("fresh_full", "exact_suffix", "stale_reuse", "cachereforge", "drift_only", "fixed_window_2")


def zero_pool(dims: dict, num_pages: int, device) -> crf.KVPool:
    """Per-layer K and V page pools of zeros, bf16 [num_pages, Hkv, 16, d]."""
    shape = (num_pages, dims["n_kv_heads"], 16, dims["head_dim"])
    return crf.KVPool([torch.zeros(shape, dtype=torch.bfloat16, device=device) for _ in range(dims["n_layers"])],
                      [torch.zeros(shape, dtype=torch.bfloat16, device=device) for _ in range(dims["n_layers"])])


class CacheState:
    """One method's cache of the prefix: K/V pages of every layer and the checkpoints H_l."""

    def __init__(self, dims: dict, n: int, num_pages: int, device):
        self.pool = zero_pool(dims, num_pages, device)
        self.H = [torch.empty(n, dims["hidden"], dtype=torch.bfloat16, device=device)
                  for _ in range(dims["n_layers"])]

    def copy_from(self, other: "CacheState") -> None:
        for a, b in zip(self.pool.k_pages + self.pool.v_pages + self.H,
                        other.pool.k_pages + other.pool.v_pages + other.H):
            a.copy_(b)


class Trajectory:
    """One prefix (``tokens`` on the pages of ``page_table``) whose adapter changes at (layer, module)."""

    def __init__(self, ctx: crf.Context, model: crf.Model, tokens: torch.Tensor, page_table: torch.Tensor,
                 layer: int, module: str, device="cuda:0"):
        dims = model.dims
        self.ctx, self.model, self.dims = ctx, model, dims
        self.n = int(tokens.shape[0])
        self.layer, self.module, self.device = layer, module, device
        self.N = dims["n_layers"]
        self.num_pages = (self.n + 15) // 16
        self.pt = page_table
        self.tokens = tokens
        self.restart = P.restart_of([(module, layer)], self.N)
        self.fin = torch.empty(dims["hidden"], dtype=torch.bfloat16, device=device)
        self.fresh_fin = torch.empty(dims["hidden"], dtype=torch.bfloat16, device=device)
        self.out_kl = torch.empty(1, dtype=torch.float32, device=device)
        self.logits = torch.empty(2, dims["vocab"], dtype=torch.float32, device=device)
        self.kl_ws = ctx.kl_workspace(1, dims["vocab"], dims["hidden"])
        self.drift_out = torch.empty(self.N, 7, 2, dtype=torch.float32, device=device)
        self._ws: Dict[Tuple[int, int, bool], torch.Tensor] = {}
        self.fresh_pool = zero_pool(dims, self.num_pages, device)

    # ------------------------------------------------------------------ device calls
    def _workspace(self, ad, req, key):
        if key not in self._ws:
            self._ws[key] = self.ctx.workspace(self.model, ad, [req])
        return self._ws[key]

    def prefill(self, ad: crf.Adapter, state: CacheState) -> None:
        req = crf.Request(self.pt, 0, self.N, n_tokens=self.n, tokens=self.tokens, hidden_out=state.H)
        self.ctx.recompute_window(self.model, ad, state.pool, [req], self._workspace(ad, req, (0, self.N, False)))

    def fresh_reference(self, ad: crf.Adapter) -> None:
        req = crf.Request(self.pt, 0, self.N, n_tokens=self.n, tokens=self.tokens, final_hidden_out=self.fresh_fin)
        self.ctx.recompute_window(self.model, ad, self.fresh_pool, [req],
                                  self._workspace(ad, req, (0, self.N, True)))

    def refresh(self, ad: crf.Adapter, state: CacheState, window: Tuple[int, int]) -> None:
        s, e = window
        if e <= s:
            return
        req = crf.Request(self.pt, s, e, n_tokens=self.n, tokens=self.tokens if s == 0 else None,
                          hidden_in=state.H[s - 1] if s > 0 else None, hidden_out=state.H[s:e])
        self.ctx.recompute_window(self.model, ad, state.pool, [req], self._workspace(ad, req, (s, e, False)))

    def first_step(self, ad: crf.Adapter, state: CacheState, window: Tuple[int, int]) -> Tuple[float, bool]:
        """KL(fresh || recovered) and top-1 agreement of the first-step distribution: the last row
        restarts from the window output (the restart state for an empty window) over this cache."""
        b = window[1] if window[1] > window[0] else window[0]
        if b == 0:
            req = crf.Request(self.pt, 0, 0, n_tokens=self.n, tokens=self.tokens, final_hidden_out=self.fin)
        else:
            req = crf.Request(self.pt, b, b, n_tokens=self.n, hidden_in=state.H[b - 1], final_hidden_out=self.fin)
        self.ctx.recompute_window(self.model, ad, state.pool, [req], self._workspace(ad, req, (b, b, True)))
        self.ctx.kl(self.model, self.fresh_fin[None], self.fin[None], self.out_kl, self.dims["vocab"], self.kl_ws,
                    logits_out=self.logits)
        top1 = bool((self.logits[0].argmax() == self.logits[1].argmax()).item())
        return float(self.out_kl.item()), top1

    def state_distance(self, vers, t: int, anchor: int, ws) -> float:
        """||theta_t - theta_anchor|| over the whole adapter state, on the device."""
        self.ctx.drift(self.model.dims_c, vers.adapter(t), [vers.adapter(anchor)] * self.N, self.drift_out, ws)
        return P.state_displacement(self.drift_out.cpu().tolist())

    # ------------------------------------------------------------------ calibration (Eq. 6-7)
    def calibrate(self, vers, versions: int, base: CacheState, scratch: CacheState, drift_ws):
        """Conditions (d_k, r, h*_k) for k = 1..versions of a calibration trajectory whose cache
        was built under version 0: h*_k is the first candidate window whose first-step state meets
        the acceptance rule against the fresh model of version k."""
        conds = []
        for k in range(1, versions + 1):
            ad = vers.adapter(k)
            self.fresh_reference(ad)
            d = self.state_distance(vers, k, 0, drift_ws)
            h_star = None
            for h in P.window_candidates(self.restart, self.N):
                scratch.copy_from(base)
                w = (self.restart, self.restart + h)
                self.refresh(ad, scratch, w)
                kl, top1 = self.first_step(ad, scratch, w)
                if kl <= KL_SAFE and top1:
                    h_star = h
                    break
            conds.append((d, self.restart, h_star if h_star is not None else self.N - self.restart))
        return conds


def drift_threshold(conds: Sequence[Tuple[float, int, int]], tail: float = 0.05) -> float:
    """The drift-only ablation's single threshold: Eq. 7's order statistic taken over the drifts of
    every calibration condition that needed recovery, pooled across layers (inf if none did)."""
    pos = sorted(d for d, _, h in conds if h > 0)
    if not pos:
        return math.inf
    return max(pos[int(math.floor(tail * len(pos)))], 1e-12)


def make_policy(method: str, n_layers: int, sens, thr) -> P.RecoveryPolicy:
    if method == "fresh_full":
        return P.RecoveryPolicy(n_layers, "full")
    if method == "exact_suffix":
        return P.RecoveryPolicy(n_layers, "suffix")
    if method == "stale_reuse":
        return P.RecoveryPolicy(n_layers, "reuse")
    if method == "cachereforge":
        return P.RecoveryPolicy(n_layers, "risk", sensitivity=sens)
    if method == "drift_only":
        return P.RecoveryPolicy(n_layers, "drift_only", threshold=thr if math.isfinite(thr) else 1e30)
    if method == "fixed_window_2":
        return P.RecoveryPolicy(n_layers, "fixed", fixed_len=2)
    raise ValueError(method)


def run(ctx, model: crf.Model, tokens: torch.Tensor, page_table: torch.Tensor, make_versions,
        versions: int = 32, calib_versions: int = 8, layer: Optional[int] = None, module: str = "v",
        methods: Sequence[str] = METHODS, device="cuda:0", calib_seed: int = 101, eval_seed: int = 202,
        sensitivity: Optional[Sequence[float]] = None, threshold: Optional[float] = None) -> dict:
    """Calibrate on one trajectory (unless ``sensitivity`` and ``threshold`` are given), then replay
    another for every method; returns the summary with each method's per-version windows and KL.
    ``make_versions(seed)`` returns that trajectory's versions: an object whose ``adapter(t)`` is
    the ``crf.Adapter`` of version t (t = 0 the adapter every cache starts from) and differs from
    version 0 only at (layer, module)."""
    n_layers = model.dims["n_layers"]
    layer = n_layers // 2 if layer is None else layer
    n = int(tokens.shape[0])
    tr = Trajectory(ctx, model, tokens, page_table, layer, module, device)
    base = CacheState(model.dims, n, tr.num_pages, device)
    conds = []
    if sensitivity is None:
        scratch = CacheState(model.dims, n, tr.num_pages, device)
        cal = make_versions(calib_seed)
        drift_ws = ctx.drift_workspace(model.dims_c, cal.adapter(0).dims_c)
        tr.prefill(cal.adapter(0), base)
        conds = tr.calibrate(cal, calib_versions, base, scratch, drift_ws)
        sens = P.calibrate_sensitivity(conds, n_layers)
        thr = drift_threshold(conds)
        del scratch, cal
    else:
        sens, thr = list(sensitivity), threshold

    ev = make_versions(eval_seed)
    drift_ws = ctx.drift_workspace(model.dims_c, ev.adapter(0).dims_c)
    tr.prefill(ev.adapter(0), base)
    states = {}
    for m in methods:
        states[m] = CacheState(model.dims, n, tr.num_pages, device)
        states[m].copy_from(base)
    del base
    pols = {m: make_policy(m, n_layers, sens, thr) for m in methods}
    stats = {m: {"maint_ms": 0.0, "kl": [], "top1": [], "frac": [], "windows": [],
                 "actions": {"reuse": 0, "bounded": 0, "suffix": 0}} for m in methods}
    ev_a, ev_b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    for t in range(1, versions + 1):
        ad = ev.adapter(t)
        tr.fresh_reference(ad)
        for m in methods:
            pol, st = pols[m], states[m]
            torch.cuda.synchronize()
            ev_a.record()
            d = ()
            if pol.mode in ("risk", "drift_only"):
                cache = {}
                for a in set(pol.anchors):
                    cache[a] = 0.0 if a == t else tr.state_distance(ev, t, a, drift_ws)
                d = [cache[a] for a in pol.anchors]
            w = pol.window(tr.restart, d)
            tr.refresh(ad, st, w)
            ev_b.record()
            torch.cuda.synchronize()
            s = stats[m]
            s["maint_ms"] += ev_a.elapsed_time(ev_b)
            pol.commit(w, t)
            kl, top1 = tr.first_step(ad, st, w)
            s["kl"].append(kl)
            s["top1"].append(top1)
            s["frac"].append(pol.fraction(w))
            s["windows"].append(list(w))
            kind = "reuse" if w[1] <= w[0] else ("suffix" if w[1] == n_layers else "bounded")
            s["actions"][kind] += 1
    ctx.check()
    out = {"calibration": {"versions": calib_versions if conds else 0, "seed": calib_seed,
                           "conditions": [{"drift": round(d, 6), "restart": r, "h_star": h} for d, r, h in conds],
                           "sensitivity_nonzero": {l: round(v, 6) for l, v in enumerate(sens) if v > 0},
                           "drift_only_threshold": thr},
           "methods": {}}
    for m in methods:
        s = stats[m]
        out["methods"][m] = {
            "maint_ms_per_trajectory": round(s["maint_ms"], 3),
            "kl_mean": sum(s["kl"]) / len(s["kl"]),
            "top1_pct": 100.0 * sum(s["top1"]) / len(s["top1"]),
            "recompute_pct": 100.0 * sum(s["frac"]) / len(s["frac"]),
            "actions": s["actions"],
            "windows": s["windows"],
            "kl": [round(v, 6) for v in s["kl"]],
        }
    return out
