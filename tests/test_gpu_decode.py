"""GPU parity of crf_decode_step: the first generated tokens on a recovered, mixed-version cache.

Two requests share a page pool; each cache is built under adapter version 0 and then recovered on
window [1, 3) under version 1, so layers hold caches of different versions. Four generation steps
follow, teacher-forced with the oracle's greedy tokens (the first from the first-step logits of the
recovered cache): at every step the device logits must match the oracle's (KL <= 1e-3), the device's
greedy token must match wherever the oracle's top-2 margin is clear, the K/V the step wrote into each
layer's page slot must match the oracle's, and every other slot of the pool stays bit-identical.
"""
import numpy as np
import pytest
import torch

import synth
from tests.harness import DeviceAdapter, DeviceModel, make_pool, pages_needed, split_page_tables
from oracle import cache as C, decoder as Dec, fidelity
from tests.gpu_util import KL_ABS, REL_KVH, oracle_adapter, oracle_model, oracle_pool, rel_frob, snapshot, to_np

pytestmark = pytest.mark.gpu

STEPS = 4


def test_decode_steps_match_oracle():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30884_gb300 as crf
    cfg, lc = synth.TINY, synth.LORA_TINY
    N = cfg.n_layers
    ns = [300, 77]
    s, e = 1, 3
    dm = DeviceModel(cfg)
    v0, v1 = DeviceAdapter(cfg, lc, 0), DeviceAdapter(cfg, lc, 1)
    P = sum(pages_needed(n + STEPS) for n in ns) + 4
    pts = split_page_tables([n + STEPS for n in ns], P, seed=6)
    pool = make_pool(cfg, P, fill="random", seed=9)
    ctx = crf.Context(0)
    opool = oracle_pool(pool)
    toks = [synth.token_ids(cfg, n, request=i, device="cuda") for i, n in enumerate(ns)]

    # GPU: stale build under v0, recovery under v1 (checkpoints kept for the window restart)
    H = [[torch.empty(n, cfg.hidden, dtype=torch.bfloat16, device="cuda") for _ in range(N)] for n in ns]
    for i, n in enumerate(ns):
        req = crf.Request(pts[i], 0, N, n_tokens=n, tokens=toks[i], hidden_out=H[i])
        ctx.recompute_window(dm.crf, v0.crf, pool, [req], ctx.workspace(dm.crf, v0.crf, [req]))
        req = crf.Request(pts[i], s, e, n_tokens=n, hidden_in=H[i][s - 1], hidden_out=H[i][s:e])
        ctx.recompute_window(dm.crf, v1.crf, pool, [req], ctx.workspace(dm.crf, v1.crf, [req]))
    ctx.check()

    # oracle: the same two steps on its own caches, then the first-step token of each request
    om, oa0, oa1 = oracle_model(dm), oracle_adapter(v0), oracle_adapter(v1)
    oreqs, first = [], []
    for i, n in enumerate(ns):
        oreq = C.RequestCache(to_np(toks[i]).astype(np.int64), pts[i].cpu().numpy())
        C.prefill(om, oa0, opool, oreq)
        _, h_last = C.recover(om, oa1, opool, oreq, s, e)
        oreqs.append(oreq)
        first.append(int(np.argmax(C.logits(om, h_last))))

    before_k, before_v = snapshot(pool)
    ws = ctx.decode_workspace(dm.crf, v1.crf, ns, pts, torch.tensor(first, dtype=torch.int32, device="cuda"))
    cur = list(first)
    for step in range(STEPS):
        pos = [n + step for n in ns]
        tok_dev = torch.tensor(cur, dtype=torch.int32, device="cuda")
        nxt = torch.empty(len(ns), dtype=torch.int32, device="cuda")
        logits = torch.empty(len(ns), cfg.vocab, dtype=torch.float32, device="cuda")
        ctx.decode_step(dm.crf, v1.crf, pool, pos, pts, tok_dev, nxt, ws, logits=logits)
        ctx.check()
        got_z, got_t = to_np(logits).astype(np.float64), to_np(nxt)
        for i in range(len(ns)):
            x = np.asarray(om.embed[cur[i]], np.float32).reshape(1, -1)
            pt = oreqs[i].page_table
            for l in range(N):
                kh, vh = opool.read(l, pt, pos[i])
                x, k, v = Dec.decode_row(x, pos[i], kh, vh, om.layers[l], oa1.layers[l], om.dims)
                opool.k[l][pt[pos[i] // 16], :, pos[i] % 16, :] = k
                opool.v[l][pt[pos[i] // 16], :, pos[i] % 16, :] = v
                page, off = int(pt[pos[i] // 16]), pos[i] % 16
                assert rel_frob(to_np(pool.k_pages[l][page, :, off, :]), k) <= REL_KVH, (step, i, l, "k")
                assert rel_frob(to_np(pool.v_pages[l][page, :, off, :]), v) <= REL_KVH, (step, i, l, "v")
            z = np.asarray(C.logits(om, x[0]), np.float64).reshape(-1)
            assert fidelity.kl(z[None], got_z[i][None])[0] <= KL_ABS, (step, i)
            top = np.sort(z)
            if top[-1] - top[-2] > 0.05:
                assert int(got_t[i]) == int(np.argmax(z)), (step, i)
            cur[i] = int(np.argmax(z))  # teacher forcing with the oracle's greedy token

    # only the generated slots changed
    written = {(int(pts[i][(n + t) // 16]), (n + t) % 16) for i, n in enumerate(ns) for t in range(STEPS)}
    for l in range(N):
        for a, b in ((pool.k_pages[l], before_k[l]), (pool.v_pages[l], before_v[l])):
            mask = torch.ones(a.shape[0], a.shape[2], dtype=torch.bool, device="cuda")
            for page, off in written:
                mask[page, off] = False
            assert torch.equal(a.permute(0, 2, 1, 3)[mask], b.permute(0, 2, 1, 3)[mask])


def test_decode_step_rejects_bad_arguments():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30884_gb300 as crf
    from paper_2609_30884_gb300.abi import CrfError
    cfg, lc = synth.TINY, synth.LORA_TINY
    dm = DeviceModel(cfg)
    ad = DeviceAdapter(cfg, lc, 1)
    P = 8
    pool = make_pool(cfg, P)
    ctx = crf.Context(0)
    pt = torch.arange(4, dtype=torch.int32, device="cuda")
    tok = torch.zeros(2, dtype=torch.int32, device="cuda")
    nxt = torch.empty(2, dtype=torch.int32, device="cuda")
    ws = ctx.decode_workspace(dm.crf, ad.crf, [20, 20], [pt, pt], tok)
    bk, bv = [t.clone() for t in pool.k_pages], [t.clone() for t in pool.v_pages]
    bad = torch.tensor([0, 99], dtype=torch.int32, device="cuda")
    logits = torch.full((2, cfg.vocab), 7.0, dtype=torch.float32, device="cuda")
    nxt.fill_(-5)
    # page tables are checked by the step's first kernel: the same page in two rows, or an id past
    # the pool, makes the step write nothing (pages, logits, tokens) and crf_check report EINVAL
    for pos, pts, t in (([20, 20], [pt, pt], tok), ([20], [bad], tok[:1])):
        ctx.decode_step(dm.crf, ad.crf, pool, pos, pts, t, nxt[:len(pos)], ws, logits=logits[:len(pos)])
        with pytest.raises(CrfError) as ei:
            ctx.check()
        assert ei.value.status == crf.abi.EINVAL
        assert all(torch.equal(a, b) for a, b in zip(pool.k_pages, bk))
        assert all(torch.equal(a, b) for a, b in zip(pool.v_pages, bv))
        assert torch.all(logits == 7.0) and torch.all(nxt == -5)
    with pytest.raises(CrfError):   # workspace too small: refused before anything is enqueued
        ctx.decode_step(dm.crf, ad.crf, pool, [20], [pt], tok[:1], nxt[:1], ws[:256])
    # a valid step on the same workspace afterwards
    ctx.decode_step(dm.crf, ad.crf, pool, [20], [pt], tok[:1], nxt[:1], ws, logits=logits[:1])
    ctx.check()
    assert not torch.all(logits[0] == 7.0) and int(nxt[0]) >= 0
