#!/usr/bin/env python3
"""Benchmark of bounded KV-cache recomputation on one GB300 per rank.

Workload (default ``7b-16k-w4``): Qwen2.5-7B-shaped random-init bf16 decoder
(28 layers, hidden 3584, 28/4 heads, SwiGLU 18944, vocab 152064), rank-16
LoRA (alpha 32) on all seven projections, one 16384-token prefix whose cache
and hidden checkpoints were built under adapter v0, current adapter v1.

One step = the whole hot path once:
  drift of v1 against every layer's anchor (28 layers x 7 modules),
  crf_recompute_window over [14, 18) from the layer-13 checkpoint (K/V
  rewritten into the permuted 16-token pages, checkpoints H_14..H_17
  refreshed), the last prefix row carried through layers 18..27 against the
  historical cache, and the first-step KL against the fresh reference.
Metric: recomputed layer*tokens/s (4 * 16384 per step). The same JSON line
carries ms per refresh for windows of 1/2/4 layers and the full prefill, the
live per-kernel roofline, an end-to-end number through pinned host buffers,
clocks, and the CPU oracle on a bounded sample.

``--impl reference`` times the CPU oracle (the plain restatement of the
method) on a bounded sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "recomputed layer*tokens/s"
UNIT = "layer*tokens/s"
# refresh sweep of the single-prefix workloads: window lengths from the workload's window start,
# and starts of complete affected suffixes (..N); full prefill is always timed. Default: 1, 2, 4.
SWEEPS = {"1.5b-16k": ((1, 2, 4, 8), (14, 26))}
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
# DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) from one ncu --set full
# capture of the kernel as it now stands, at the full launch size of the 7B-shape 16K workload
# (profiles/gemm_gateup_swiglu_7b16k.md). An entry is removed whenever its kernel changes.
NCU_TRAFFIC_BYTES = {"gemm_gateup_swiglu": 2.921001e9 + 0.616805e9}


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return p, "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                 "-i", str(self.index), "-lms", "100", "-f", self.path],
                stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        with open(self.path) as f:
            lines = f.readlines()
        os.unlink(self.path)
        return self.summarise(lines)

    @staticmethod
    def summarise(lines):
        """Median SM clock, the maximum clock and the throttle reasons seen Active in the
        nvidia-smi CSV rows of the query above."""
        rows = []
        for line in lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 9:
                rows.append(parts)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = set()
        sm = []
        for r in rows:
            try:
                sm.append(float(r[1]))
            except ValueError:
                pass
            for j, nm in enumerate(names):
                if r[5 + j].lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": float(rows[0][2]) if rows[0][2].replace(".", "").isdigit() else None,
                "samples": len(rows), "reasons": sorted(reasons)}


# ----------------------------------------------------------------------------- ranks
def max_over_ranks(x: float, device="cpu") -> float:
    """The largest value of x over all ranks (x itself without a process group)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank: float, steps: int, world: int, max_ms: float) -> float:
    """Whole-job rate: every rank's units over the slowest rank's time."""
    return world * units_per_rank * steps / (max_ms / 1000.0)


# ----------------------------------------------------------------------------- workload
def algorithmic_work(cfg, lc, n):
    """Algorithmic FLOPs per kernel kind for one recomputed layer over n tokens (and bytes).

    Each projection counts its base product, the adapter's down products x A^T (2 n r in per
    adapted module) and its up products (2 n r out), all computed in the same launch.
    """
    h, f, qd, kvd, r = cfg.hidden, cfg.ffn, cfg.n_q_heads * cfg.head_dim, cfg.n_kv_heads * cfg.head_dim, lc.rank
    ad = lambda m: m in lc.modules
    lora = lambda m, i, out: 2 * n * r * (i + out) if ad(m) else 0
    flops = {
        "gemm_qkv_rope_paged": 2 * n * h * (qd + 2 * kvd) + lora("q", h, qd) + lora("k", h, kvd) + lora("v", h, kvd),
        "gemm_o_resid": 2 * n * qd * h + lora("o", qd, h),
        "gemm_gateup_swiglu": 2 * n * h * 2 * f + lora("gate", h, f) + lora("up", h, f),
        "gemm_down_resid": 2 * n * f * h + lora("down", f, h),
        "attn_prefill_paged": 4 * cfg.n_q_heads * cfg.head_dim * n * (n + 1) // 2,
    }
    byts = {"rmsnorm": 2 * (2 * n * h * 2)}   # two norms, read + write bf16
    return flops, byts


def step_bytes(cfg, lc, ns, wins):
    """Algorithmic HBM bytes of the step's bandwidth-bound parts, once per step.

    drift_gram: both adapter versions' factors of every layer and module (bf16). tail_decode: per
    request, the weights of layers e..N-1 (base rows and LoRA A and B, bf16) and the K/V of its
    prefix at those layers. lm_head: the head's rows once (fresh and recovered rows share the pass).
    """
    h, f, qd, kvd, r = cfg.hidden, cfg.ffn, cfg.n_q_heads * cfg.head_dim, cfg.n_kv_heads * cfg.head_dim, lc.rank
    dims = {"q": (h, qd), "k": (h, kvd), "v": (h, kvd), "o": (qd, h), "gate": (h, f), "up": (h, f), "down": (f, h)}
    lora = sum(r * (i + o) * 2 for m, (i, o) in dims.items() if m in lc.modules)
    base = sum(i * o * 2 for i, o in dims.values())
    tail = sum((cfg.n_layers - e) * (base + lora + 2 * (n - 1) * kvd * 2) for n, (_, e) in zip(ns, wins))
    return {"drift_gram": 2 * cfg.n_layers * lora, "tail_decode": tail,
            "lm_head": cfg.vocab * h * 2}


def shard_requests(loads, world):
    """Split independent requests over ranks (longest first onto the least-loaded rank).

    Returns one list of request indices per rank; with a single request every rank gets it
    (independent replicas).
    """
    if len(loads) == 1:
        return [[0] for _ in range(world)]
    order = sorted(range(len(loads)), key=lambda i: -loads[i])
    bins = [[] for _ in range(world)]
    tot = [0.0] * world
    for i in order:
        r = min(range(world), key=lambda k: (tot[k], k))
        bins[r].append(i)
        tot[r] += loads[i]
    return [sorted(b) for b in bins]


def build_state(wl, device, ctx, rank=0, world=1):
    """Model, adapters, stale cache, checkpoints and the step's requests for this rank's share.

    Every request's cache and checkpoints are built by a stale prefill under its own older
    adapter version (current - gap); its fresh reference final row by a prefill under the
    current version. Only the checkpoints the window reads or rewrites are kept.
    """
    import torch
    import synth
    import paper_2609_30884_gb300 as crf
    from tests.harness import DeviceAdapter, DeviceModel, make_pool, split_page_tables

    cfg, lc = wl.model, wl.lora
    N = cfg.n_layers
    loads = [(e - s) * n for n, (s, e) in zip(wl.n_tokens, wl.windows)]
    mine = shard_requests(loads, world)[rank]
    ns = [wl.n_tokens[i] for i in mine]
    wins = [wl.windows[i] for i in mine]
    cur_v = wl.cur_version
    stale_v = [cur_v - wl.stale_gap[i] for i in mine]
    dm = DeviceModel(cfg, device)
    versions = {v: DeviceAdapter(cfg, lc, v, device) for v in sorted(set(stale_v) | {cur_v})}
    v_cur = versions[cur_v]
    P = sum((n + 15) // 16 for n in ns)
    pool = make_pool(cfg, P, device)
    pts = split_page_tables(ns, P, seed=1, device=device)
    R = len(mine)
    fin = torch.empty(R, cfg.hidden, dtype=torch.bfloat16, device=device)
    fresh = torch.empty(R, cfg.hidden, dtype=torch.bfloat16, device=device)
    # size the workspace for the largest of the set-up prefills and the batched step
    prefills = [crf.Request(pts[k], 0, N, n_tokens=ns[k], final_hidden_out=fresh[k]) for k in range(R)]
    step_reqs0 = [crf.Request(pts[k], wins[k][0], wins[k][1], n_tokens=ns[k], final_hidden_out=fin[k])
                  for k in range(R)]
    ws_bytes = max(ctx.workspace_size(dm.crf, v_cur.crf, [r]) for r in prefills)
    ws_bytes = max(ws_bytes, ctx.workspace_size(dm.crf, v_cur.crf, step_reqs0))
    ws = torch.empty(ws_bytes + 256, dtype=torch.uint8, device=device)
    tokens, h_in, h_out, reqs = [], [], [], []
    for k in range(R):
        n, (s, e) = ns[k], wins[k]
        tok = synth.token_ids(cfg, n, request=mine[k], device=device)
        ctx.recompute_window(dm.crf, v_cur.crf, pool,
                             [crf.Request(pts[k], 0, N, tokens=tok, final_hidden_out=fresh[k])], ws)
        ck = [torch.empty(n, cfg.hidden, dtype=torch.bfloat16, device=device) for _ in range(N)]
        ctx.recompute_window(dm.crf, versions[stale_v[k]].crf, pool,
                             [crf.Request(pts[k], 0, N, tokens=tok, hidden_out=ck)], ws)
        torch.cuda.synchronize()
        tokens.append(tok)
        h_in.append(ck[s - 1] if s > 0 else None)
        h_out.append(ck[s:e])
        reqs.append(crf.Request(pts[k], s, e, n_tokens=n, tokens=tok, hidden_in=h_in[k],
                                hidden_out=h_out[k], final_hidden_out=fin[k]))
        del ck
    ctx.check()
    # each layer's anchor: the stale version of the first request whose window covers it
    anchor_v = []
    for l in range(N):
        cover = [k for k in range(R) if wins[k][0] <= l < wins[k][1]]
        anchor_v.append(stale_v[cover[0] if cover else 0])
    st = {"cfg": cfg, "lc": lc, "mine": mine, "ns": ns, "wins": wins, "dm": dm,
          "versions": versions, "v_cur": v_cur, "pool": pool, "pts": pts, "tokens": tokens,
          "h_in": h_in, "h_out": h_out, "reqs": reqs, "ws": ws, "fin": fin, "fresh": fresh,
          "anchors": [versions[v].crf for v in anchor_v],
          "out_sq": torch.empty(N, 7, 2, dtype=torch.float32, device=device),
          "dws": ctx.drift_workspace(dm.crf.dims_c, v_cur.crf.dims_c),
          "out_kl": torch.empty(R, dtype=torch.float32, device=device),
          "kws": ctx.kl_workspace(R, cfg.vocab, cfg.hidden),
          "units": sum((e - s) * n for n, (s, e) in zip(ns, wins))}
    return st


def run_step(ctx, st, reqs=None):
    ctx.drift(st["dm"].crf.dims_c, st["v_cur"].crf, st["anchors"], st["out_sq"], st["dws"])
    ctx.recompute_window(st["dm"].crf, st["v_cur"].crf, st["pool"], reqs or st["reqs"], st["ws"])
    ctx.kl(st["dm"].crf, st["fresh"], st["fin"], st["out_kl"], st["cfg"].vocab, st["kws"])


def second_input_set(st):
    """A second set of restart buffers and the same requests reading them, so that the host
    copy of one step's inputs can run while the previous step computes."""
    import torch
    import paper_2609_30884_gb300 as crf
    h_in2 = [torch.empty_like(h) if h is not None else None for h in st["h_in"]]
    reqs2 = []
    for k, r in enumerate(st["reqs"]):
        s, e = st["wins"][k]
        reqs2.append(crf.Request(st["pts"][k], s, e, n_tokens=st["ns"][k], tokens=st["tokens"][k],
                                 hidden_in=h_in2[k], hidden_out=st["h_out"][k],
                                 final_hidden_out=st["fin"][k]))
    return h_in2, reqs2


def time_refresh(ctx, st, s, e, reps=3):
    """ms of crf_recompute_window alone for window [s, e) (no tail decode)."""
    import torch
    import paper_2609_30884_gb300 as crf
    n = st["ns"][0]
    w0 = st["wins"][0]
    # the window's restart state is the layer s-1 checkpoint; rewrite into scratch outputs
    import torch as _t
    if s == 0:
        hin = None
    elif s == w0[0]:
        hin = st["h_in"][0]
    elif w0[0] <= s - 1 < w0[1]:
        hin = st["h_out"][0][s - 1 - w0[0]]
    else:
        hin = st["h_in"][0]  # a stand-in restart state: the refresh's cost does not depend on its values
    outs = [_t.empty(n, st["cfg"].hidden, dtype=_t.bfloat16, device=st["fin"].device)
            for _ in range(e - s)]
    req = crf.Request(st["pts"][0], s, e, n_tokens=n, tokens=st["tokens"][0], hidden_in=hin,
                      hidden_out=outs)
    ctx.recompute_window(st["dm"].crf, st["v_cur"].crf, st["pool"], [req], st["ws"])
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(reps):
        ctx.recompute_window(st["dm"].crf, st["v_cur"].crf, st["pool"], [req], st["ws"])
    b.record()
    torch.cuda.synchronize()
    return a.elapsed_time(b) / reps


# ----------------------------------------------------------------------------- CPU oracle
def cpu_oracle_sample(wl, n_rows, layer=None, x=None, weights=None, adapter=None):
    """Time the oracle on one window layer over the first n_rows tokens of the prefix."""
    import numpy as np
    import synth
    from oracle import build as obuild, decoder as D
    cfg, lc = wl.model, wl.lora
    layer = wl.windows[0][0] if layer is None else layer
    P = obuild.layer_params(cfg, layer, tensors=weights)
    A = obuild.layer_adapter(cfg, lc, 1, layer, tensors=adapter)
    if x is None:
        x = synth.hidden_state(cfg, n_rows, "bench_restart", layer).float().numpy()
    dims = obuild.dims_of(cfg)
    t0 = time.perf_counter()
    D.decoder_layer(np.asarray(x[:n_rows], np.float32), P, A, dims, np.float32, chunk=512)
    return time.perf_counter() - t0


def blas_threads():
    try:
        from threadpoolctl import threadpool_info
        return max((i.get("num_threads", 0) for i in threadpool_info()), default=os.cpu_count())
    except Exception:
        return int(os.environ.get("OPENBLAS_NUM_THREADS", os.cpu_count() or 1))


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    import synth
    wl = workload_of(args)
    n_rows = args.ref_rows
    s, _ = wl.windows[0]
    weights = synth.layer_weights(wl.model, s)
    adapter = synth.adapter_version(wl.model, wl.lora, 1, s)
    import numpy as np
    x = synth.hidden_state(wl.model, n_rows, "bench_restart", s).float().numpy()
    for _ in range(args.warmup):
        cpu_oracle_sample(wl, n_rows, s, x, weights, adapter)
    times = [cpu_oracle_sample(wl, n_rows, s, x, weights, adapter) for _ in range(args.steps)]
    ms = 1000.0 * statistics.mean(times)
    value = n_rows / (ms / 1000.0)
    cores = blas_threads()
    sample = (f"oracle decoder layer {s} of {wl.name} over the first {n_rows} of "
              f"{wl.n_tokens[0]} tokens per step (fp32 NumPy); an upper bound on the oracle's rate "
              f"over the whole prefix, whose later rows attend to more keys")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": f"synthetic (seeded counter-based generator, random-init {wl.model.name})",
            "config": config_of(wl),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def config_of(wl):
    cfg = {"workload": f"{args_workload_name(wl)}: {wl.name}", "n_layers": wl.model.n_layers,
           "lora_rank": wl.lora.rank, "lora_modules": list(wl.lora.modules), "page_tokens": 16,
           "l2": "inputs larger than L2 (window weights of >= 466 MB per layer per step)"}
    if len(wl.n_tokens) == 1:
        s, e = wl.windows[0]
        cfg.update(prefix_tokens=wl.n_tokens[0], window=[s, e], layers_recomputed=e - s)
    else:
        cfg.update(requests=len(wl.n_tokens), prefix_tokens=list(wl.n_tokens),
                   windows=[list(w) for w in wl.windows], stale_gaps=list(wl.stale_gap),
                   layer_tokens=sum((e - s) * n for n, (s, e) in zip(wl.n_tokens, wl.windows)))
    return cfg


def args_workload_name(wl):
    import synth
    for k, v in synth.WORKLOADS.items():
        if v is wl:
            return k
    return wl.name


def run_window_only(args):
    """One window layer (or a few) over the prefix, nothing else: the small profiling case.

    Holds only the window's layer weights, one KV pool and the workspace (a few GB for the
    7B shape), so a kernel of the window can be captured by a profiler on its own.
    """
    import torch
    import synth
    import paper_2609_30884_gb300 as crf
    from tests.harness import DeviceAdapter, DeviceModel, make_pool, pages_needed

    wl = workload_of(args)
    cfg, lc = wl.model, wl.lora
    n = args.tokens or wl.n_tokens[0]
    s, e = wl.windows[0]
    device = "cuda:0"
    ctx = crf.Context(0)
    dm = DeviceModel(cfg, device, layers=range(s, e), with_head=False)
    cur = DeviceAdapter(cfg, lc, 1, device, layers=range(s, e))
    P = pages_needed(n)
    pool = make_pool(cfg, P, device)
    pt = synth.page_permutation(P, 1, device)
    h_in = synth.hidden_state(cfg, n, device=device)
    h_out = [torch.empty(n, cfg.hidden, dtype=torch.bfloat16, device=device) for _ in range(e - s)]
    req = crf.Request(pt, s, e, hidden_in=h_in, hidden_out=h_out)
    ws = ctx.workspace(dm.crf, cur.crf, [req])
    for _ in range(args.warmup):
        ctx.recompute_window(dm.crf, cur.crf, pool, [req], ws)
    ctx.check()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(args.steps):
        ctx.recompute_window(dm.crf, cur.crf, pool, [req], ws)
    b.record()
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / args.steps
    ctx.profile_enable(True, 4096)
    for _ in range(args.steps):
        ctx.recompute_window(dm.crf, cur.crf, pool, [req], ws)
    prof = ctx.profile_read()
    ctx.profile_enable(False)
    flops, _ = algorithmic_work(cfg, lc, n)
    kern = {}
    for k, (kms, cnt) in prof.items():
        if k == "_dropped" or cnt == 0:
            continue
        kern[k] = {"ms_per_window": round(kms / args.steps, 4)}
        if k in flops:
            kern[k]["tflops"] = round(flops[k] * (e - s) * args.steps / (kms / 1000.0) / 1e12, 1)
    print(json.dumps({"case": "window-only", "workload": args.workload, "tokens": n,
                      "window": [s, e], "ms_per_window": ms,
                      "layer_tokens_per_s": (e - s) * n / (ms / 1000.0), "kernels": kern}))
    ctx.close()
    return 0


def run_decode_only(args):
    """The last layer as the window and its last row through the tail: the small profiling case
    of the decode-row kernels (layers N-2, N-1 of the workload's shape, one KV pool)."""
    import torch
    import synth
    import paper_2609_30884_gb300 as crf
    from tests.harness import DeviceAdapter, DeviceModel, make_pool, pages_needed, split_page_tables

    wl = workload_of(args)
    cfg, lc = wl.model, wl.lora
    n = args.tokens or wl.n_tokens[0]
    s, e = cfg.n_layers - 2, cfg.n_layers - 1
    device = "cuda:0"
    ctx = crf.Context(0)
    dm = DeviceModel(cfg, device, layers=range(s, cfg.n_layers), with_head=False)
    cur = DeviceAdapter(cfg, lc, 1, device, layers=range(s, cfg.n_layers))
    P = pages_needed(n)
    pool = make_pool(cfg, P, device, fill="random", seed=11)
    pt = split_page_tables([n], P, seed=5, device=device)[0]
    h_in = synth.hidden_state(cfg, n, "restart", s - 1, device=device)
    fin = torch.empty(cfg.hidden, dtype=torch.bfloat16, device=device)
    req = crf.Request(pt, s, e, hidden_in=h_in, final_hidden_out=fin)
    ws = ctx.workspace(dm.crf, cur.crf, [req])
    for _ in range(args.warmup):
        ctx.recompute_window(dm.crf, cur.crf, pool, [req], ws)
    ctx.check()
    ctx.profile_enable(True, 4096)
    for _ in range(args.steps):
        ctx.recompute_window(dm.crf, cur.crf, pool, [req], ws)
    prof = ctx.profile_read()
    ctx.profile_enable(False)
    ctx.check()
    kern = {k: {"ms_per_call": round(kms / args.steps, 4), "launches": cnt // args.steps}
            for k, (kms, cnt) in prof.items() if k != "_dropped" and cnt}
    print(json.dumps({"case": "decode-only", "workload": args.workload, "tokens": n,
                      "window": [s, e], "tail_layers": cfg.n_layers - e, "kernels": kern}))
    ctx.close()
    return 0


def run_trajectory_case(args):
    """The recovery policy over a synthetic 32-version adapter trajectory (RQ4-style)."""
    import torch
    import paper_2609_30884_gb300 as crf
    from paper_2609_30884_gb300 import trajectory
    from tests.harness import DeviceModel, Versions, pages_needed, split_page_tables

    wl = workload_of(args)
    cfg, lc = wl.model, wl.lora
    n = args.tokens or wl.n_tokens[0]
    ctx = crf.Context(0)
    dm = DeviceModel(cfg, "cuda:0")
    layer = args.update_layer if args.update_layer >= 0 else cfg.n_layers // 2
    pt = split_page_tables([n], pages_needed(n), seed=1, device="cuda:0")[0]
    t0 = time.time()
    res = trajectory.run(ctx, dm.crf, synth_tokens(cfg, n), pt,
                         lambda seed: Versions(cfg, lc, layer, args.update_module, args.update_std, seed,
                                               "cuda:0", 0),
                         versions=args.versions, calib_versions=args.calib_versions, layer=layer,
                         module=args.update_module)
    line = {"case": "trajectory", "workload": f"{args.workload}: {wl.name}", "tokens": n,
            "versions": args.versions,
            "update": {"layer": layer, "module": args.update_module, "std_per_entry": args.update_std,
                       "version_0": "the workload adapter before any perturbation (A ~ N(0, 0.02^2), "
                                    "B ~ N(0, 0.01^2))",
                       "factors": "A and B, every entry, one seeded N(0, std^2) step per version"},
            "maintenance": "crf_drift queries + crf_recompute_window of the chosen window (+ host decision), "
                           "CUDA events, summed over the versions",
            "data": "synthetic (seeded random-init decoder, uniform token ids)",
            "wall_s": round(time.time() - t0, 1), **res}
    print(json.dumps(line))
    ctx.close()
    return 0


def run_tail_case(args):
    """Offline tail-influence sweep: N + 1 hybrid first-step passes over a stale cache."""
    import torch
    import numpy as np
    import paper_2609_30884_gb300 as crf
    from paper_2609_30884_gb300 import tail
    from tests.harness import DeviceModel, Versions, make_pool, pages_needed, split_page_tables

    wl = workload_of(args)
    cfg, lc = wl.model, wl.lora
    n = args.tokens or wl.n_tokens[0]
    N = cfg.n_layers
    layer = args.update_layer if args.update_layer >= 0 else N // 2
    ctx = crf.Context(0)
    dm = DeviceModel(cfg, "cuda:0")
    vers = Versions(cfg, lc, layer, args.update_module, args.update_std, 202, "cuda:0", 0)
    old, cur = vers.adapter(0), vers.adapter(args.versions)
    P = pages_needed(n)
    pt = split_page_tables([n], P, seed=1, device="cuda:0")[0]
    tokens = synth_tokens(cfg, n)
    stale, fresh = make_pool(cfg, P, "cuda:0"), make_pool(cfg, P, "cuda:0")
    H = [torch.empty(n, cfg.hidden, dtype=torch.bfloat16, device="cuda:0") for _ in range(N)]
    for ad, pool, hid in ((old, stale, None), (cur, fresh, H)):
        req = crf.Request(pt, 0, N, n_tokens=n, tokens=tokens, hidden_out=hid)
        ctx.recompute_window(dm.crf, ad, pool, [req], ctx.workspace(dm.crf, ad, [req]))
    tail.sweep(ctx, dm.crf, cur, stale, pt, n, tokens, H, cfg.vocab)   # warm-up
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    a.record()
    rows = torch.empty(N + 1, cfg.hidden, dtype=torch.bfloat16, device="cuda:0")
    tail.hybrid_rows(ctx, dm.crf, cur, stale, pt, n, tokens, H, rows)
    b.record()
    torch.cuda.synchronize()
    ms_rows = a.elapsed_time(b)
    res = tail.sweep(ctx, dm.crf, cur, stale, pt, n, tokens, H, cfg.vocab)
    r = layer
    print(json.dumps({
        "case": "tail-influence", "workload": f"{args.workload}: {wl.name}", "tokens": n,
        "update": {"layer": layer, "module": args.update_module, "std_per_entry": args.update_std,
                   "versions": args.versions},
        "ms_hybrid_rows": round(ms_rows, 3), "hybrid_passes": N + 1,
        "kl": [round(float(x), 6) for x in res.kl], "tail_T": [round(float(x), 4) for x in res.tail],
        "margin": round(res.margin, 4), "top1": [bool(x) for x in res.top1],
        "kl_certificate_holds": int(res.kl_certificate_holds.sum()),
        "top1_certificate_holds": int(res.top1_certificate_holds.sum()),
        "horizon_eps_0.05": res.horizon(r, 0.05),
        "data": "synthetic (seeded random-init decoder, uniform token ids)"}))
    ctx.close()
    return 0


def run_decode_case(args):
    """Greedy generation on the paged cache: R requests of the workload's prefix length, T steps."""
    import torch
    import paper_2609_30884_gb300 as crf
    import synth
    from tests.harness import DeviceAdapter, DeviceModel, make_pool, pages_needed, split_page_tables

    wl = workload_of(args)
    cfg, lc = wl.model, wl.lora
    n = args.tokens or wl.n_tokens[0]
    R, T = args.decode_rows, args.decode_steps
    N = cfg.n_layers
    ctx = crf.Context(0)
    dm = DeviceModel(cfg, "cuda:0")
    ad = DeviceAdapter(cfg, lc, wl.cur_version, "cuda:0")
    P = R * pages_needed(n + T + args.warmup)
    pts = split_page_tables([n + T + args.warmup] * R, P, seed=1, device="cuda:0")
    pool = make_pool(cfg, P, "cuda:0")
    for i in range(R):
        tok = synth.token_ids(cfg, n, request=i, device="cuda:0")
        req = crf.Request(pts[i], 0, N, n_tokens=n, tokens=tok)
        ctx.recompute_window(dm.crf, ad.crf, pool, [req], ctx.workspace(dm.crf, ad.crf, [req]))
    cur = synth.token_ids(cfg, R, request=99, device="cuda:0")
    nxt = torch.empty(R, dtype=torch.int32, device="cuda:0")
    pos = [n] * R
    ws = ctx.decode_workspace(dm.crf, ad.crf, [n + T + args.warmup] * R, pts, cur)
    for _ in range(args.warmup):
        ctx.decode_step(dm.crf, ad.crf, pool, pos, pts, cur, nxt, ws)
        cur, nxt = nxt, cur
        pos = [p_ + 1 for p_ in pos]
    ctx.check()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    a.record()
    for _ in range(T):
        ctx.decode_step(dm.crf, ad.crf, pool, pos, pts, cur, nxt, ws)
        cur, nxt = nxt, cur
        pos = [p_ + 1 for p_ in pos]
    b.record()
    torch.cuda.synchronize()
    ctx.check()
    ms = a.elapsed_time(b)
    h, f, qd, kvd, V = cfg.hidden, cfg.ffn, cfg.n_q_heads * cfg.head_dim, cfg.n_kv_heads * cfg.head_dim, cfg.vocab
    w_bytes = 2 * N * (h * (qd + 2 * kvd) + qd * h + 2 * h * f + f * h) + 2 * V * h
    kv_bytes = sum(2 * N * 2 * kvd * (p_ - T // 2) for p_ in pos)   # mean cached length over the run
    step_ms = ms / T
    peaks, src = load_peaks()
    gbs = (w_bytes + kv_bytes) / (step_ms / 1000.0) / 1e9
    print(json.dumps({"case": "decode", "workload": f"{args.workload}: {wl.name}", "prefix_tokens": n,
                      "rows": R, "steps": T, "ms_per_step": round(step_ms, 3),
                      "tokens_per_s": round(R * T / (ms / 1000.0), 1),
                      "hbm": {"bytes_per_step": w_bytes + kv_bytes, "achieved_gbs": round(gbs, 1),
                              "peak_gbs": peaks["hbm_gbs"], "frac": round(gbs / peaks["hbm_gbs"], 4),
                              "peak_source": src},
                      "data": "synthetic (seeded random-init decoder, uniform token ids)"}))
    ctx.close()
    return 0


def run_drift_case(args):
    """crf_drift alone (every layer and module of the workload's adapter against a per-layer anchor):
    the small profiling case of the drift kernels (adapters only on the device)."""
    import torch
    import paper_2609_30884_gb300 as crf
    from tests.harness import DeviceAdapter, DeviceModel

    wl = workload_of(args)
    cfg, lc = wl.model, wl.lora
    ctx = crf.Context(0)
    dm = DeviceModel(cfg, "cuda:0", layers=[], with_head=False)
    cur = DeviceAdapter(cfg, lc, 3, "cuda:0")
    anchors = [DeviceAdapter(cfg, lc, v, "cuda:0") for v in (0, 1, 2)]
    which = [anchors[l % 3].crf for l in range(cfg.n_layers)]
    out = torch.empty(cfg.n_layers, 7, 2, dtype=torch.float32, device="cuda:0")
    ws = ctx.drift_workspace(dm.crf.dims_c, cur.crf.dims_c)
    for _ in range(args.warmup):
        ctx.drift(dm.crf.dims_c, cur.crf, which, out, ws)
    ctx.check()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    # the device sleeps while the host enqueues every timed call, so the events time the device
    # alone (a call's host side, ctypes marshalling and two launches, can outlast its kernels)
    torch.cuda._sleep(int(2e6) * max(1, args.steps))
    a.record()
    h0 = time.perf_counter()
    for _ in range(args.steps):
        ctx.drift(dm.crf.dims_c, cur.crf, which, out, ws)
    host_us = (time.perf_counter() - h0) / args.steps * 1e6
    b.record()
    torch.cuda.synchronize()
    ctx.check()
    ms = a.elapsed_time(b) / args.steps
    factor_bytes = 0
    for l in range(cfg.n_layers):
        for m, (A, B) in cur.layers[l].items():
            factor_bytes += 2 * (A.numel() + B.numel()) * 2   # both versions, bf16
    peaks, src = load_peaks()
    gbs = factor_bytes / (ms / 1000.0) / 1e9
    print(json.dumps({"case": "drift", "workload": f"{args.workload}: {wl.name}", "rank": lc.rank,
                      "modules": list(lc.modules), "ms_per_call": round(ms, 4),
                      "host_us_per_call": round(host_us, 1),
                      "hbm": {"bytes": factor_bytes, "achieved_gbs": round(gbs, 1),
                              "frac": round(gbs / peaks["hbm_gbs"], 4), "peak_source": src}}))
    ctx.close()
    return 0


def run_kl_only(args):
    """crf_kl with the model's head alone (final norm + LM head GEMV + KL over --decode-rows row
    pairs): the small profiling case of the head kernels (only the head weights on the device)."""
    import torch
    import synth
    import paper_2609_30884_gb300 as crf
    from tests.harness import DeviceModel

    wl = workload_of(args)
    cfg = wl.model
    rows = max(1, args.decode_rows)
    ctx = crf.Context(0)
    dm = DeviceModel(cfg, "cuda:0", layers=[], with_head=True)
    h_ref = synth.hidden_state(cfg, rows, "kl_ref", device="cuda:0")
    h_cur = synth.hidden_state(cfg, rows, "kl_cur", device="cuda:0")
    out = torch.empty(rows, dtype=torch.float32, device="cuda:0")
    ws = ctx.kl_workspace(rows, cfg.vocab, cfg.hidden)
    for _ in range(args.warmup):
        ctx.kl(dm.crf, h_ref, h_cur, out, cfg.vocab, ws)
    ctx.check()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(args.steps):
        ctx.kl(dm.crf, h_ref, h_cur, out, cfg.vocab, ws)
    b.record()
    torch.cuda.synchronize()
    ctx.check()
    ms = a.elapsed_time(b) / args.steps
    head_bytes = cfg.vocab * cfg.hidden * 2
    peaks, src = load_peaks()
    print(json.dumps({"case": "kl-only", "workload": f"{args.workload}: {wl.name}", "row_pairs": rows,
                      "ms_per_call": round(ms, 4),
                      "hbm": {"bytes": head_bytes, "achieved_gbs": round(head_bytes / (ms / 1000.0) / 1e9, 1),
                              "frac": round(head_bytes / (ms / 1000.0) / 1e9 / peaks["hbm_gbs"], 4),
                              "peak_source": src}}))
    ctx.close()
    return 0


def synth_tokens(cfg, n):
    import synth
    return synth.token_ids(cfg, n, device="cuda:0")


def workload_of(args):
    """The named workload, with the adapter's rank / modules replaced when the flags ask for it
    (alpha / r stays 2, as in the specified configurations)."""
    import synth
    from dataclasses import replace
    wl = synth.workload(args.workload)
    if args.lora_rank or args.lora_modules:
        rank = args.lora_rank or wl.lora.rank
        mods = tuple(args.lora_modules.split(",")) if args.lora_modules else wl.lora.modules
        wl = replace(wl, lora=replace(wl.lora, rank=rank, alpha=2.0 * rank, modules=mods))
    return wl


# ----------------------------------------------------------------------------- main
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="crf", choices=["crf", "reference"])
    ap.add_argument("--workload", default="7b-16k-w4")
    ap.add_argument("--cpu-rows", type=int, default=4096, help="tokens in the CPU-oracle sample")
    ap.add_argument("--ref-rows", type=int, default=1024, help="tokens per reference-arm step")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-sweep", action="store_true")
    ap.add_argument("--case", default="step",
                    choices=["step", "window-only", "decode-only", "trajectory", "tail-influence", "decode",
                             "drift", "kl-only"],
                    help="window-only / decode-only: small profiling cases (window layers only / "
                         "the last layer and its first-step row); trajectory: the recovery policy "
                         "over a synthetic continual-adapter trajectory; tail-influence: the offline "
                         "N + 1 hybrid-pass sweep (the update and --versions as for trajectory)")
    ap.add_argument("--versions", type=int, default=32, help="trajectory: adapter updates replayed")
    ap.add_argument("--decode-rows", type=int, default=8,
                    help="decode: requests generating together; kl-only: row pairs")
    ap.add_argument("--decode-steps", type=int, default=32, help="decode: timed generation steps")
    ap.add_argument("--calib-versions", type=int, default=8, help="trajectory: calibration updates")
    ap.add_argument("--update-layer", type=int, default=-1, help="trajectory: updated layer (-1: N // 2)")
    ap.add_argument("--update-module", default="v", help="trajectory: updated module")
    ap.add_argument("--update-std", type=float, default=0.1, help="trajectory: step std per entry")
    ap.add_argument("--tokens", type=int, default=0, help="prefix length for --case window-only")
    ap.add_argument("--lora-rank", type=int, default=0, help="adapter rank override (4, 8 or 16)")
    ap.add_argument("--lora-modules", default="",
                    help="adapter modules override, comma separated (e.g. v or q,v)")
    args = ap.parse_args()
    if args.case == "window-only":
        return run_window_only(args)
    if args.case == "decode-only":
        return run_decode_only(args)
    if args.case == "trajectory":
        return run_trajectory_case(args)
    if args.case == "tail-influence":
        return run_tail_case(args)
    if args.case == "decode":
        return run_decode_case(args)
    if args.case == "drift":
        return run_drift_case(args)
    if args.case == "kl-only":
        return run_kl_only(args)
    if args.warmup < 3 and args.impl == "crf":
        args.warmup = 3
    if args.impl == "reference":
        return run_reference(args)

    import torch
    import torch.distributed as dist

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device(f"cuda:{local}"))
    torch.cuda.set_device(local)
    device = f"cuda:{local}"

    from paper_2609_30884_gb300 import build as _build
    if rank == 0 or world == 1:
        _build.build()
    if world > 1:
        dist.barrier()
    import synth
    import paper_2609_30884_gb300 as crf

    wl = workload_of(args)
    cfg, lc = wl.model, wl.lora
    ctx = crf.Context(local)
    st = build_state(wl, device, ctx, rank, world)
    n, (s, e) = st["ns"][0], st["wins"][0]
    units = st["units"]

    for _ in range(args.warmup):
        run_step(ctx, st)
    ctx.check()

    # ---------------- timed region: device-resident inputs. The step time comes from a loop with
    # nothing else on the stream; the per-kernel times (roofline) from a second loop of the same
    # steps with the library's CUDA events around every launch, which add a few microseconds of
    # gap per launch.
    clocks = ClockSampler(local)
    clocks.start()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(args.steps):
        run_step(ctx, st)
    t1.record()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    elapsed_ms = t0.elapsed_time(t1)
    ctx.profile_enable(True, 8192)
    p0, p1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    p0.record()
    for _ in range(args.steps):
        run_step(ctx, st)
    p1.record()
    torch.cuda.synchronize()
    profiled_ms_step = p0.elapsed_time(p1) / args.steps
    prof = ctx.profile_read()
    ctx.profile_enable(False)
    clk = clocks.stop()
    ctx.check()
    elapsed_ms = max_over_ranks(elapsed_ms, device)
    ms_step = elapsed_ms / args.steps
    value = job_throughput(units, args.steps, world, elapsed_ms)

    # ---------------- end to end: restart state from pinned host memory, KL back to host.
    # Every step's restart state crosses from pinned host memory inside the timed region; the
    # copy for step i + 1 runs on a copy stream into the other of two buffer sets while step i
    # computes (events order each buffer's copy after the compute that last read it).
    h_host = [h.to("cpu").pin_memory() if h is not None else None for h in st["h_in"]]
    kl_host = torch.empty(st["out_kl"].numel(), dtype=torch.float32).pin_memory()
    stream = torch.cuda.current_stream()
    copy_stream = torch.cuda.Stream(device=device)
    h_in2, reqs2 = second_input_set(st)
    sets = [(st["h_in"], st["reqs"]), (h_in2, reqs2)]

    def e2e_run(steps, start):
        copied = [torch.cuda.Event(), torch.cuda.Event()]
        done = [None, None]

        def copy_into(i):
            with torch.cuda.stream(copy_stream):
                if done[i % 2] is not None:
                    copy_stream.wait_event(done[i % 2])
                for h_dev, hh in zip(sets[i % 2][0], h_host):
                    if hh is not None:
                        h_dev.copy_(hh, non_blocking=True)
                copied[i % 2].record(copy_stream)

        copy_stream.wait_event(start)
        copy_into(0)
        for i in range(steps):
            stream.wait_event(copied[i % 2])
            if i + 1 < steps:
                copy_into(i + 1)
            run_step(ctx, st, sets[i % 2][1])
            ev = torch.cuda.Event()
            ev.record(stream)
            done[i % 2] = ev
            kl_host.copy_(st["out_kl"], non_blocking=True)

    warm = torch.cuda.Event()
    warm.record(stream)
    e2e_run(2, warm)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    e2e_run(args.steps, a)
    b.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(a.elapsed_time(b), device)
    h2d = sum(h.numel() * 2 for h in st["h_in"] if h is not None)
    e2e = {"value": job_throughput(units, args.steps, world, e2e_ms), "unit": UNIT,
           "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": 4 * kl_host.numel(),
           "ms_per_step": e2e_ms / args.steps,
           "kl_first_step": [round(float(v), 6) for v in kl_host.tolist()]}

    # ---------------- per-kernel roofline from the live events
    peaks, peak_src = load_peaks()
    # algorithmic work of one step: per request, (e - s) layers over its own prefix length
    flops_step, bytes_step = {}, {}
    for n_i, (s_i, e_i) in zip(st["ns"], st["wins"]):
        fl, by = algorithmic_work(cfg, lc, n_i)
        for k, v in fl.items():
            flops_step[k] = flops_step.get(k, 0) + v * (e_i - s_i)
        for k, v in by.items():
            bytes_step[k] = bytes_step.get(k, 0) + v * (e_i - s_i)
    for k, v in step_bytes(cfg, lc, st["ns"], st["wins"]).items():
        bytes_step[k] = bytes_step.get(k, 0) + v
    flops_layer, _ = algorithmic_work(cfg, lc, n)
    kernels = {}
    gpu_launches = 0
    for name, (ms, cnt) in prof.items():
        if name == "_dropped":
            continue
        gpu_launches += cnt
        entry = {"launches": cnt, "ms_total": round(ms, 4),
                 "ms_per_step": round(ms / args.steps, 4)}
        if name in flops_step:
            fl = flops_step[name] * args.steps
            tf = fl / (ms / 1000.0) / 1e12
            entry.update(bound="tensor", tflops=round(tf, 1),
                         frac=round(tf / peaks["bf16_tflops"], 4))
        if name in bytes_step:
            by = bytes_step[name] * args.steps
            gbs = by / (ms / 1000.0) / 1e9
            entry.update(bound="hbm", gbs=round(gbs, 1), frac=round(gbs / peaks["hbm_gbs"], 4))
        kernels[name] = entry
    dom = max((k for k in kernels if k in flops_step), key=lambda k: kernels[k]["ms_total"])
    launches_dom = kernels[dom]["launches"]
    roofline = {"kernel": dom, "bound": "tensor", "achieved": kernels[dom]["tflops"],
                "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                "frac": kernels[dom]["frac"],
                "traffic": NCU_TRAFFIC_BYTES.get(dom) if wl.model.hidden == 3584 and n == 16384 else None,
                "peak_source": f"bf16_tflops ({peak_src}, burst)",
                "frac_of_sustained": round(kernels[dom]["tflops"] / peaks.get("bf16_tflops_sustained", 1700.0), 4),
                "algorithmic_flops_per_launch": flops_step[dom] / max(1, kernels[dom]["launches"] // args.steps),
                "launches": launches_dom}
    gemm_names = [k for k in kernels if k.startswith("gemm_") and k in flops_step]
    gemm_fl = sum(flops_step[k] for k in gemm_names) * args.steps
    gemm_ms = sum(kernels[k]["ms_total"] for k in gemm_names)
    gemm_tf = gemm_fl / (gemm_ms / 1000.0) / 1e12 if gemm_ms else 0.0

    # ---------------- window sweep (ms per 16K-prefix refresh)
    sweep = {}
    if not args.no_sweep and len(st["ns"]) == 1:
        lengths, suffix_starts = SWEEPS.get(args.workload, ((1, 2, 4), ()))
        for ln in lengths:
            sweep[f"window_{ln}"] = round(time_refresh(ctx, st, s, min(s + ln, cfg.n_layers)), 3)
        for s0 in suffix_starts:
            sweep[f"suffix_{s0}_{cfg.n_layers}"] = round(time_refresh(ctx, st, s0, cfg.n_layers, reps=2), 3)
        sweep["full_prefill_28"] = round(time_refresh(ctx, st, 0, cfg.n_layers, reps=2), 3)
        sweep["layer_tokens_per_s_full"] = round(cfg.n_layers * n / (sweep["full_prefill_28"] / 1000.0))

    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": f"synthetic (seeded counter-based generator, random-init {wl.model.name})",
            "config": config_of(wl), "gpu_launches": gpu_launches, "e2e": e2e,
            "roofline": roofline, "clocks": clk,
            "gemm_tflops_all": round(gemm_tf, 1),
            "gemm_frac_all": round(gemm_tf / peaks["bf16_tflops"], 4),
            "ms_per_refresh": sweep, "kernels": kernels,
            "kernels_timing": ("CUDA events around every library launch, in a second loop of the "
                               "same steps after the timed one: %.3f ms/step with the events" %
                               profiled_ms_step),
            "step": ("drift(N x 7) + crf_recompute_window over every request's window (rows of "
                     "requests active at a layer batched) + tail decode of each last row through "
                     "layers e..N-1 + first-step KL per request")}

    # ---------------- CPU oracle baseline (rank 0, one GPU only)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        w = {k: v.to("cpu") for k, v in st["dm"].layers[s].items()}
        ad = {m: (a.to("cpu"), b.to("cpu")) for m, (a, b) in st["v_cur"].layers[s].items()}
        x = st["h_in"][0][:args.cpu_rows].float().cpu().numpy() if s > 0 else None
        secs = cpu_oracle_sample(wl, args.cpu_rows, s, x, w, ad)
        line["cpu_baseline"] = {
            "value": args.cpu_rows / secs, "unit": UNIT, "cores": blas_threads(), "kind": "oracle",
            "sample": (f"oracle decoder layer {s} over the first {args.cpu_rows} of {n} tokens "
                       f"(fp32 NumPy), {secs:.1f} s; an upper bound on the oracle's rate over the "
                       f"whole prefix, whose later rows attend to more keys")}
    if rank == 0:
        print(json.dumps(line))
    ctx.close()
    if world > 1:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
