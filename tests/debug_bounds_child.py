"""Run in a child process by tests/test_gpu_bounds.py with CRF_LIB_VARIANT=debug and
CRF_DEBUG_DEVICE_CHECKS_ONLY=1: the CRF_DEBUG library, whose page-table check at the start of each call is skipped,
so its device-side checks alone meet the bad page ids below.

1. A valid two-request prefill matches the oracle and records nothing (no false positives).
2. Out-of-range page ids (one past the pool, negative) in a prefill, in a window whose final row
   decodes through the historical pages, and in a generation step (a page that is only read, the
   page the step writes): each is reported as CRF_EINVAL, and the report is cleared.
3. The context still computes the valid prefill to the oracle's values afterwards.
"""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

import synth  # noqa: E402
import paper_2609_30884_gb300 as crf  # noqa: E402
from tests.harness import DeviceAdapter, DeviceModel, make_pool, pages_needed, split_page_tables  # noqa: E402
from oracle import cache as C  # noqa: E402
from tests.gpu_util import (REL_KVH, oracle_adapter, oracle_model, oracle_pool, rel_frob,  # noqa: E402
                            request_kv, to_np)


def expect_bounds_error(ctx, what):
    try:
        ctx.check()
    except crf.CrfError as e:
        assert e.status == crf.abi.EINVAL, (what, str(e))
        assert "page id" in str(e), (what, str(e))
    else:
        raise AssertionError(f"{what}: bad page id not reported")
    ctx.check()  # cleared


def valid_prefill(ctx, dm, ad, om, oa, cfg):
    ns = [100, 37]
    P = sum(pages_needed(n) for n in ns) + 3
    pts = split_page_tables(ns, P, seed=8)
    pool = make_pool(cfg, P, fill="random", seed=4)
    opool = oracle_pool(pool)
    toks = [synth.token_ids(cfg, n, request=i, device="cuda") for i, n in enumerate(ns)]
    reqs = [crf.Request(pts[i], 0, cfg.n_layers, tokens=toks[i]) for i in range(len(ns))]
    ctx.recompute_window(dm.crf, ad.crf, pool, reqs, ctx.workspace(dm.crf, ad.crf, reqs))
    ctx.check()
    for i, n in enumerate(ns):
        oreq = C.RequestCache(to_np(toks[i]).astype(np.int64), pts[i].cpu().numpy())
        C.prefill(om, oa, opool, oreq)
        for l in range(cfg.n_layers):
            err = rel_frob(request_kv(pool.k_pages[l], pts[i], n),
                           request_kv(torch.from_numpy(opool.k[l]), pts[i], n))
            assert err <= REL_KVH, (i, l, err)


def main():
    assert crf.abi.LIB_PATH.endswith("libcrf_debug.so"), crf.abi.LIB_PATH
    torch.cuda.set_device(0)
    cfg, lc = synth.TINY, synth.LORA_TINY
    N = cfg.n_layers
    dm = DeviceModel(cfg)
    ad = DeviceAdapter(cfg, lc, 1)
    om, oa = oracle_model(dm), oracle_adapter(ad)
    ctx = crf.Context(0)
    ctx.check()

    valid_prefill(ctx, dm, ad, om, oa, cfg)

    n = 70
    P = pages_needed(n) + 2
    toks = synth.token_ids(cfg, n, request=3, device="cuda")
    for bad in (P, -1):
        # prefill: the bad page is written by the QKV epilogue and read by the attention
        pool = make_pool(cfg, P, fill="random", seed=5)
        pt = split_page_tables([n], P, seed=2)[0].clone()
        pt[2] = bad
        req = crf.Request(pt, 0, N, tokens=toks)
        ctx.recompute_window(dm.crf, ad.crf, pool, [req], ctx.workspace(dm.crf, ad.crf, [req]))
        expect_bounds_error(ctx, f"prefill, page id {bad}")

        # window [1, 2) whose final row decodes through layers 2..N-1 over the historical pages
        pool = make_pool(cfg, P, fill="random", seed=6)
        pt = split_page_tables([n], P, seed=2)[0].clone()
        pt[1] = bad
        h_in = synth.hidden_state(cfg, n, device="cuda")
        fin = torch.empty(cfg.hidden, dtype=torch.bfloat16, device="cuda")
        req = crf.Request(pt, 1, 2, hidden_in=h_in, final_hidden_out=fin)
        ctx.recompute_window(dm.crf, ad.crf, pool, [req], ctx.workspace(dm.crf, ad.crf, [req]))
        expect_bounds_error(ctx, f"window with tail, page id {bad}")

        # generation step at position 40: page 0 of the table is read, page 2 is written
        pool = make_pool(cfg, 8, fill="random", seed=7)
        nxt = torch.empty(1, dtype=torch.int32, device="cuda")
        t = torch.tensor([5], dtype=torch.int32, device="cuda")
        for slot in (0, 2):
            ids = [3, 6, 1]
            ids[slot] = bad if bad >= 0 else -1
            if bad == P:
                ids[slot] = 8       # one past this pool
            pts = [torch.tensor(ids, dtype=torch.int32, device="cuda")]
            ws = ctx.decode_workspace(dm.crf, ad.crf, [40], pts, t)
            ctx.decode_step(dm.crf, ad.crf, pool, [40], pts, t, nxt, ws)
            expect_bounds_error(ctx, f"decode, table slot {slot}")

    valid_prefill(ctx, dm, ad, om, oa, cfg)
    ctx.close()
    print("debug bounds ok")


if __name__ == "__main__":
    main()
