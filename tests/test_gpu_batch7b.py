"""GPU parity of the batched 7B-shape workload: 8 cached prefixes of 2K-16K tokens, each with
its own window, one shared pool with a randomly permuted page table.

* Batching is invisible in the window: the batched call gives bit-identical pages and refreshed
  checkpoints to running every request alone (each row is computed the same way whatever else
  shares its tile or launch); the first-step rows agree to the per-layer 1e-2 bar (their GEMV
  kernel depends on how many rows share a weight pass, and its rounding compounds over the layers
  after the window).
* Against the oracle, per request, on what it computes at this size: K and V of every position of
  the request's first window layer, and that layer's output at 48 rows spread over the prefix,
  held to 1e-2 or 1.25x the distance the oracle's layer moves at the same rows when it stores its
  intermediates in bf16 where the path does, whichever is larger. Deep layers of an adapter
  several versions old are adapter-dominated: attention scores have a spread of ~1e3 and top-2
  gaps of a few units, so a rounding-sized change flips which key a head attends to. Windows
  starting at layer 3 or below are well conditioned and meet the plain 1e-2 bar.
* Slots no request owns, and layers outside every window, stay bit-identical.
"""
import numpy as np
import pytest
import torch

import synth
from tests.harness import DeviceAdapter, DeviceModel, make_pool, split_page_tables
from oracle import build as obuild, decoder as Dec
from tests.gpu_util import (REL_KVH, STORAGE_FACTOR, bf16_storage_rows, free_slots, rel_frob, snapshot,
                            to_np, untouched_mask)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30884_gb300 as crf
    return crf.Context(0)


def _requests(crf, cfg, wl, pts):
    reqs, keep = [], []
    for i, (n, (s, e)) in enumerate(zip(wl.n_tokens, wl.windows)):
        tok = synth.token_ids(cfg, n, request=i, device="cuda")
        h_in = synth.hidden_state(cfg, n, "restart", 100 + i, device="cuda") if s > 0 else None
        h_out = [torch.empty(n, cfg.hidden, dtype=torch.bfloat16, device="cuda") for _ in range(e - s)]
        fin = torch.empty(cfg.hidden, dtype=torch.bfloat16, device="cuda")
        reqs.append(crf.Request(pts[i], s, e, n_tokens=n, tokens=tok, hidden_in=h_in,
                                hidden_out=h_out, final_hidden_out=fin))
        keep.append((tok, h_in, h_out, fin))
    return reqs, keep


def test_batch7b_equals_single_and_oracle(ctx):
    import paper_2609_30884_gb300 as crf
    wl = synth.workload("7b-batch8")
    cfg = wl.model
    dm = DeviceModel(cfg)
    cur = DeviceAdapter(cfg, wl.lora, wl.cur_version)
    P = sum((n + 15) // 16 for n in wl.n_tokens) + 11
    pts = split_page_tables(wl.n_tokens, P, seed=1)
    pool = make_pool(cfg, P, fill="random", seed=13)
    bk, bv = snapshot(pool)

    reqs, keep = _requests(crf, cfg, wl, pts)
    ctx.recompute_window(dm.crf, cur.crf, pool, reqs, ctx.workspace(dm.crf, cur.crf, reqs))
    ctx.check()
    got_k = [t.clone() for t in pool.k_pages]
    got_v = [t.clone() for t in pool.v_pages]

    # every request alone on a fresh copy of the historical pool
    fin_err = []
    for i in range(len(reqs)):
        for l in range(cfg.n_layers):
            pool.k_pages[l].copy_(bk[l])
            pool.v_pages[l].copy_(bv[l])
        one, keep1 = _requests(crf, cfg, wl, pts)
        ctx.recompute_window(dm.crf, cur.crf, pool, [one[i]], ctx.workspace(dm.crf, cur.crf, [one[i]]))
        ctx.check()
        s, e = wl.windows[i]
        n = wl.n_tokens[i]
        for l in range(s, e):
            assert torch.equal(request_kv_t(pool.k_pages[l], pts[i], n), request_kv_t(got_k[l], pts[i], n)), (i, l)
            assert torch.equal(request_kv_t(pool.v_pages[l], pts[i], n), request_kv_t(got_v[l], pts[i], n)), (i, l)
            assert torch.equal(keep1[i][2][l - s], keep[i][2][l - s]), (i, l)
        # the first-step row takes the tensor-core GEMV (main and adapter-down products) when >= 3
        # rows share a weight pass and the CUDA-core one alone: both fp32-accurate, but their
        # rounding differs and compounds over every layer the row passes after its window (26 after a
        # window [0, 2)), so it is held to the per-layer bar the oracle tests use
        fin_err.append(rel_frob(to_np(keep1[i][3]), to_np(keep[i][3])))
    print("first-step row, batched vs alone:", [f"{x:.2e}" for x in fin_err])
    assert max(fin_err) <= REL_KVH, fin_err

    # untouched slots and layers, bit-exact
    free = untouched_mask(P, list(zip(pts, wl.n_tokens)))
    covered = {l for (s, e) in wl.windows for l in range(s, e)}
    for l in range(cfg.n_layers):
        if l in covered:
            assert torch.equal(free_slots(got_k[l], free), free_slots(bk[l], free))
            assert torch.equal(free_slots(got_v[l], free), free_slots(bv[l], free))
        else:
            assert torch.equal(got_k[l], bk[l]) and torch.equal(got_v[l], bv[l])

    # oracle: first window layer of every request
    dims = obuild.dims_of(cfg)
    for i, (n, (s, e)) in enumerate(zip(wl.n_tokens, wl.windows)):
        P_l = obuild.layer_params(cfg, s, tensors=dm.layers[s])
        A_l = obuild.layer_adapter(cfg, wl.lora, wl.cur_version, s, tensors=cur.layers[s])
        tok, h_in, h_out, _ = keep[i]
        x = to_np(h_in) if s > 0 else to_np(dm.embed[tok.long()])
        q_all, k_all, v_all = Dec.qkv(x, P_l, A_l, dims, np.arange(n))
        rows = np.unique(np.concatenate([[0, 15, 16, n - 2, n - 1], np.linspace(32, n - 3, 43).astype(int)]))
        st_h, st_k, st_v = bf16_storage_rows(x, P_l, A_l, dims, rows)
        want = []
        for t in rows:
            o = Dec.single_query_attention(q_all[t], k_all[:t + 1], v_all[:t + 1])
            want.append(Dec.post_attention(x[t:t + 1], o[None], P_l, A_l, dims)[0])
        want = np.stack(want)
        got = to_np(h_out[0])[rows]
        report = [("k", rel_frob(to_np(request_kv_t(got_k[s], pts[i], n)), k_all), rel_frob(st_k, k_all)),
                  ("v", rel_frob(to_np(request_kv_t(got_v[s], pts[i], n)), v_all), rel_frob(st_v, v_all)),
                  ("h", rel_frob(got, want), rel_frob(st_h, want))]
        print(f"request {i} n={n} window [{s},{e}) first layer (name, err, bf16-storage distance):",
              [(a, round(b, 5), round(c, 5)) for a, b, c in report])
        for name, err, dist in report:
            assert err <= max(REL_KVH, STORAGE_FACTOR * dist), (i, name, err, dist)
            if s <= 3:   # the shallowest windows are well conditioned: the plain bar
                assert err <= REL_KVH, (i, name, err)


def request_kv_t(pool_layer, page_table, n):
    """Rows of positions 0..n-1 of one request from a pool layer [P, Hkv, 16, d] (device tensor)."""
    t = torch.arange(n, device=pool_layer.device)
    pages = page_table.to(pool_layer.device).long()[t // 16]
    return pool_layer[pages, :, t % 16, :]
