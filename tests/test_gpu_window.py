"""GPU parity of crf_recompute_window against the oracle on the same seeded inputs."""
import numpy as np
import pytest
import torch

import synth
from tests.harness import DeviceAdapter, DeviceModel, make_pool, pages_needed, split_page_tables
from oracle import cache as C
from tests.gpu_util import (REL_KVH, free_slots, oracle_adapter, oracle_model, oracle_pool,
                            rel_frob, request_kv, snapshot, to_np, untouched_mask)

pytestmark = pytest.mark.gpu

torch_cuda = pytest.importorskip("torch.cuda")


@pytest.fixture(scope="module")
def ctx():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30884_gb300 as crf
    return crf.Context(0)


@pytest.fixture(scope="module")
def tiny():
    cfg, lc = synth.TINY, synth.LORA_TINY
    dm = DeviceModel(cfg)
    cur = DeviceAdapter(cfg, lc, 1)
    return cfg, lc, dm, cur, oracle_model(dm), oracle_adapter(cur)


def _run(ctx, dm, ad, pool, reqs):
    ws = ctx.workspace(dm.crf, ad.crf, reqs)
    ctx.recompute_window(dm.crf, ad.crf, pool, reqs, ws)
    ctx.check()


def _check_request(cfg, pool, before, opool, pt, n, s, e, h_out, o_hidden, tag=""):
    for l in range(s, e):
        for which, gp, op in (("k", pool.k_pages, opool.k), ("v", pool.v_pages, opool.v)):
            got = request_kv(gp[l], pt, n)
            want = request_kv(torch.from_numpy(op[l]), pt, n)
            err = rel_frob(got, want)
            assert err <= REL_KVH, f"{tag} layer {l} {which}: rel err {err:.3e}"
        if h_out is not None:
            err = rel_frob(to_np(h_out[l - s]), o_hidden[l])
            assert err <= REL_KVH, f"{tag} layer {l} hidden: rel err {err:.3e}"


@pytest.mark.parametrize("n,s,e", [(512, 2, 4), (512, 1, 2), (300, 0, 2), (512, 2, 2),
                                   (17, 1, 3), (1, 0, 4), (129, 3, 4)])
def test_window_single_request(ctx, tiny, n, s, e):
    cfg, lc, dm, cur, om, oa = tiny
    P = pages_needed(n) + 7
    pool = make_pool(cfg, P, fill="random", seed=5)
    pt = split_page_tables([n], P, seed=3)[0]
    tokens = synth.token_ids(cfg, n, device="cuda")
    h_in = synth.hidden_state(cfg, n, device="cuda") if s > 0 else None
    h_out = [torch.empty(n, cfg.hidden, dtype=torch.bfloat16, device="cuda") for _ in range(e - s)]
    fin = torch.empty(cfg.hidden, dtype=torch.bfloat16, device="cuda")
    bk, bv = snapshot(pool)
    opool = oracle_pool(pool)
    import paper_2609_30884_gb300 as crf
    req = crf.Request(pt, s, e, n_tokens=n, tokens=tokens, hidden_in=h_in,
                      hidden_out=h_out if e > s else None, final_hidden_out=fin)
    _run(ctx, dm, cur, pool, [req])

    oreq = C.RequestCache(to_np(tokens).astype(np.int64), pt.cpu().numpy())
    restart = to_np(h_in) if s > 0 else None
    _, h_last = C.recover(om, oa, opool, oreq, s, e, restart=restart)

    _check_request(cfg, pool, (bk, bv), opool, pt, n, s, e, h_out if e > s else None, oreq.hidden)
    # bit-exact: layers outside the window, and slots the request does not own
    free = untouched_mask(P, [(pt, n)])
    for l in range(cfg.n_layers):
        if s <= l < e:
            assert torch.equal(free_slots(pool.k_pages[l], free), free_slots(bk[l], free))
            assert torch.equal(free_slots(pool.v_pages[l], free), free_slots(bv[l], free))
        else:
            assert torch.equal(pool.k_pages[l], bk[l])
            assert torch.equal(pool.v_pages[l], bv[l])
    err = rel_frob(to_np(fin), h_last)
    assert err <= REL_KVH, f"final hidden rel err {err:.3e}"


def test_batched_requests_shared_pool(ctx, tiny):
    cfg, lc, dm, cur, om, oa = tiny
    lengths = [100, 257, 512]
    windows = [(0, 2), (1, 4), (2, 3)]
    P = sum(pages_needed(n) for n in lengths) + 9
    pool = make_pool(cfg, P, fill="random", seed=6)
    pts = split_page_tables(lengths, P, seed=4)
    bk, bv = snapshot(pool)
    opool = oracle_pool(pool)
    import paper_2609_30884_gb300 as crf
    reqs, keep = [], []
    for i, (n, (s, e)) in enumerate(zip(lengths, windows)):
        tokens = synth.token_ids(cfg, n, request=i, device="cuda")
        h_in = synth.hidden_state(cfg, n, layer=i, device="cuda") if s > 0 else None
        h_out = [torch.empty(n, cfg.hidden, dtype=torch.bfloat16, device="cuda") for _ in range(e - s)]
        fin = torch.empty(cfg.hidden, dtype=torch.bfloat16, device="cuda")
        reqs.append(crf.Request(pts[i], s, e, n_tokens=n, tokens=tokens, hidden_in=h_in,
                                hidden_out=h_out, final_hidden_out=fin))
        keep.append((tokens, h_in, h_out, fin))
    _run(ctx, dm, cur, pool, reqs)
    for i, (n, (s, e)) in enumerate(zip(lengths, windows)):
        tokens, h_in, h_out, fin = keep[i]
        oreq = C.RequestCache(to_np(tokens).astype(np.int64), pts[i].cpu().numpy())
        _, h_last = C.recover(om, oa, opool, oreq, s, e,
                              restart=to_np(h_in) if s > 0 else None)
        _check_request(cfg, pool, (bk, bv), opool, pts[i], n, s, e, h_out, oreq.hidden, tag=f"req{i}")
        assert rel_frob(to_np(fin), h_last) <= REL_KVH
    free = untouched_mask(P, list(zip(pts, lengths)))
    for l in range(cfg.n_layers):
        assert torch.equal(free_slots(pool.k_pages[l], free), free_slots(bk[l], free))
        assert torch.equal(free_slots(pool.v_pages[l], free), free_slots(bv[l], free))


def test_identical_adapter_reproduces_stale_cache_bitexact(ctx, tiny):
    cfg, lc, dm, _, _, _ = tiny
    v0 = DeviceAdapter(cfg, lc, 0)
    n = 300
    P = pages_needed(n) + 2
    pool = make_pool(cfg, P)
    pt = split_page_tables([n], P, seed=8)[0]
    tokens = synth.token_ids(cfg, n, device="cuda")
    hs = [torch.empty(n, cfg.hidden, dtype=torch.bfloat16, device="cuda") for _ in range(cfg.n_layers)]
    import paper_2609_30884_gb300 as crf
    _run(ctx, dm, v0, pool, [crf.Request(pt, 0, cfg.n_layers, tokens=tokens, hidden_out=hs)])
    bk, bv = snapshot(pool)
    h2 = [torch.empty_like(hs[0]) for _ in range(2)]
    _run(ctx, dm, v0, pool, [crf.Request(pt, 1, 3, hidden_in=hs[0], hidden_out=h2)])
    for l in range(cfg.n_layers):
        assert torch.equal(pool.k_pages[l], bk[l]) and torch.equal(pool.v_pages[l], bv[l])
    assert torch.equal(h2[0], hs[1]) and torch.equal(h2[1], hs[2])


def test_query_only_update_one_layer_window_keeps_kv(ctx, tiny):
    """Eq. S4: a query-only update at layer s, window [s, s+1), rewrites K/V bit-identically."""
    cfg, lc, dm, _, _, _ = tiny
    v0 = DeviceAdapter(cfg, lc, 0)
    s = 1
    A, B = v0.layers[s]["q"]
    vq = DeviceAdapter(cfg, lc, 0, override={(s, "q"): ((A.float() + 0.05).bfloat16(),
                                                         (B.float() - 0.05).bfloat16())})
    n = 200
    P = pages_needed(n)
    pool = make_pool(cfg, P)
    pt = split_page_tables([n], P, seed=9)[0]
    tokens = synth.token_ids(cfg, n, device="cuda")
    hs = [torch.empty(n, cfg.hidden, dtype=torch.bfloat16, device="cuda") for _ in range(cfg.n_layers)]
    import paper_2609_30884_gb300 as crf
    _run(ctx, dm, v0, pool, [crf.Request(pt, 0, cfg.n_layers, tokens=tokens, hidden_out=hs)])
    bk, bv = snapshot(pool)
    h_new = [torch.empty_like(hs[0])]
    _run(ctx, dm, vq, pool, [crf.Request(pt, s, s + 1, hidden_in=hs[s - 1], hidden_out=h_new)])
    for l in range(cfg.n_layers):
        assert torch.equal(pool.k_pages[l], bk[l]) and torch.equal(pool.v_pages[l], bv[l])
    assert not torch.equal(h_new[0], hs[s])


def test_full_prefill_matches_oracle_prefill(ctx, tiny):
    """Window [0, N) from the embedding is a fresh prefill; compared layer by layer."""
    cfg, lc, dm, cur, om, oa = tiny
    n = 384
    P = pages_needed(n)
    pool = make_pool(cfg, P)
    pt = split_page_tables([n], P, seed=10)[0]
    tokens = synth.token_ids(cfg, n, request=3, device="cuda")
    hs = [torch.empty(n, cfg.hidden, dtype=torch.bfloat16, device="cuda") for _ in range(cfg.n_layers)]
    fin = torch.empty(cfg.hidden, dtype=torch.bfloat16, device="cuda")
    import paper_2609_30884_gb300 as crf
    _run(ctx, dm, cur, pool, [crf.Request(pt, 0, cfg.n_layers, tokens=tokens, hidden_out=hs,
                                          final_hidden_out=fin)])
    opool = C.PagedPool(cfg.n_layers, P, cfg.n_kv_heads, cfg.head_dim)
    oreq = C.RequestCache(to_np(tokens).astype(np.int64), pt.cpu().numpy())
    x = C.prefill(om, oa, opool, oreq)
    for l in range(cfg.n_layers):
        assert rel_frob(to_np(hs[l]), oreq.hidden[l]) <= REL_KVH
        assert rel_frob(request_kv(pool.k_pages[l], pt, n), request_kv(torch.from_numpy(opool.k[l]), pt, n)) <= REL_KVH
        assert rel_frob(request_kv(pool.v_pages[l], pt, n), request_kv(torch.from_numpy(opool.v[l]), pt, n)) <= REL_KVH
    assert rel_frob(to_np(fin), x[-1]) <= REL_KVH


def test_invalid_arguments_rejected(ctx, tiny):
    """Host-checkable arguments are refused before anything is enqueued (CRF_EINVAL / CRF_ENOMEM)."""
    cfg, lc, dm, cur, _, _ = tiny
    import paper_2609_30884_gb300 as crf
    n = 64
    P = pages_needed(n)
    pool = make_pool(cfg, P)
    pt = split_page_tables([n], P, seed=2)[0]
    h = synth.hidden_state(cfg, n, device="cuda")
    ws = torch.empty(1 << 24, dtype=torch.uint8, device="cuda")
    bk, _ = snapshot(pool)
    bad = [
        crf.Request(pt, 3, 2, hidden_in=h),                      # s > e
        crf.Request(pt, 1, 5, hidden_in=h),                      # e > N
        crf.Request(pt, 1, 2, n_tokens=n),                       # missing hidden_in
        crf.Request(pt, 2, 2, hidden_in=h),                      # empty window, no final out
    ]
    for r in bad:
        with pytest.raises(crf.CrfError) as ei:
            ctx.recompute_window(dm.crf, cur.crf, pool, [r], ws)
        assert ei.value.status == crf.abi.EINVAL
    with pytest.raises(crf.CrfError) as ei:
        ctx.recompute_window(dm.crf, cur.crf, pool, [crf.Request(pt, 1, 2, hidden_in=h)], ws[:1024])
    assert ei.value.status == crf.abi.ENOMEM
    torch.cuda.synchronize()
    assert all(torch.equal(a, b) for a, b in zip(pool.k_pages, bk))


def test_bad_page_tables_rejected_on_device(ctx, tiny):
    """Page ids are checked by the first kernel of the call, without a host round trip: an id
    outside the pool, a page used twice within a request or shared by two requests, makes the
    call write nothing outside its workspace (pool, checkpoints, final rows) and crf_check report
    CRF_EINVAL once; the next call with valid tables runs normally."""
    cfg, lc, dm, cur, om, oa = tiny
    import paper_2609_30884_gb300 as crf
    n = 64
    P = 2 * pages_needed(n)
    pool = make_pool(cfg, P, fill="random", seed=4)
    pt0, pt1 = split_page_tables([n, n], P, seed=2)
    h = synth.hidden_state(cfg, n, device="cuda")
    ws = torch.empty(1 << 24, dtype=torch.uint8, device="cuda")
    bk, bv = snapshot(pool)
    hout = [torch.full((n, cfg.hidden), 3.0, dtype=torch.bfloat16, device="cuda")]
    fin = torch.full((cfg.hidden,), 5.0, dtype=torch.bfloat16, device="cuda")
    shared = pt1.clone()
    shared[1] = pt0[2]
    cases = [
        [crf.Request(torch.full_like(pt0, P), 1, 2, hidden_in=h, hidden_out=hout, final_hidden_out=fin)],
        [crf.Request(torch.full_like(pt0, -1), 1, 2, hidden_in=h, hidden_out=hout)],
        [crf.Request(torch.zeros_like(pt0), 1, 2, hidden_in=h, hidden_out=hout, final_hidden_out=fin)],
        [crf.Request(pt0, 1, 2, hidden_in=h, hidden_out=hout),
         crf.Request(shared, 1, 3, hidden_in=h, final_hidden_out=fin)],
        [crf.Request(torch.full_like(pt0, P), 3, 4, hidden_in=h, final_hidden_out=fin)],   # last layer
    ]
    for reqs in cases:
        ctx.recompute_window(dm.crf, cur.crf, pool, reqs, ws)    # enqueued: nothing waits here
        with pytest.raises(crf.CrfError) as ei:
            ctx.check()
        assert ei.value.status == crf.abi.EINVAL
        ctx.check()                                                # reported once
        assert all(torch.equal(a, b) for a, b in zip(pool.k_pages, bk))
        assert all(torch.equal(a, b) for a, b in zip(pool.v_pages, bv))
        assert torch.all(hout[0] == 3.0) and torch.all(fin == 5.0)
    # the same workspace then serves a valid call
    _run(ctx, dm, cur, pool, [crf.Request(pt0, 1, 2, hidden_in=h, hidden_out=hout, final_hidden_out=fin)])
    assert not torch.equal(pool.k_pages[1], bk[1])
    assert not torch.all(hout[0] == 3.0)
