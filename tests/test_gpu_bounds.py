"""Device-side bounds checks, exercised without a fault: every bad id is caught before it is used
as an address, replaced by a safe one (token 0, page 0), recorded in the context's status word and
reported by crf_check as CRF_EINVAL; the report is cleared and the context keeps working.

Token ids are checked in every build. Page ids are checked by the first kernel of every call
(which rejects the whole call); the library built with CRF_DEBUG (libcrf_debug.so) re-checks them
at every device-side use, and with CRF_DEBUG_DEVICE_CHECKS_ONLY=1 it skips that first check so that
the per-use checks alone meet the bad ids. That build runs in a child process
(tests/debug_bounds_child.py)."""
import os
import subprocess
import sys

import pytest
import torch

import synth
from tests.harness import DeviceAdapter, DeviceModel, make_pool, pages_needed, split_page_tables

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def test_bad_token_id_is_reported_and_read_as_token_zero():
    _need_gpu()
    import paper_2609_30884_gb300 as crf
    cfg, lc = synth.TINY, synth.LORA_TINY
    N, n = cfg.n_layers, 40
    dm = DeviceModel(cfg)
    ad = DeviceAdapter(cfg, lc, 1)
    P = pages_needed(n) + 2
    pt = split_page_tables([n], P, seed=4)[0]
    ctx = crf.Context(0)
    ctx.check()
    toks = synth.token_ids(cfg, n, request=0, device="cuda")
    bad = toks.clone()
    bad[7] = cfg.vocab             # one past the vocabulary
    bad[23] = -3
    good = toks.clone()
    good[7] = 0
    good[23] = 0

    outs = []
    for t, expect_error in ((bad, True), (good, False)):
        pool = make_pool(cfg, P, fill="random", seed=2)
        fin = torch.empty(cfg.hidden, dtype=torch.bfloat16, device="cuda")
        req = crf.Request(pt, 0, N, tokens=t, final_hidden_out=fin)
        ctx.recompute_window(dm.crf, ad.crf, pool, [req], ctx.workspace(dm.crf, ad.crf, [req]))
        if expect_error:
            with pytest.raises(crf.CrfError) as ei:
                ctx.check()
            assert ei.value.status == crf.abi.EINVAL
            assert "token id" in str(ei.value)
        ctx.check()                # cleared, and nothing else recorded
        outs.append((pool, fin))
    # the bad ids were read as token 0: both runs wrote the same pages and the same final row
    (pb, fb), (pg, fg) = outs
    assert torch.equal(fb, fg)
    for l in range(N):
        assert torch.equal(pb.k_pages[l], pg.k_pages[l]) and torch.equal(pb.v_pages[l], pg.v_pages[l])


def test_bad_decode_token_is_reported():
    _need_gpu()
    import paper_2609_30884_gb300 as crf
    cfg, lc = synth.TINY, synth.LORA_TINY
    dm = DeviceModel(cfg)
    ad = DeviceAdapter(cfg, lc, 1)
    pool = make_pool(cfg, 8, fill="random", seed=3)
    ctx = crf.Context(0)
    pts = [torch.tensor([5, 2], dtype=torch.int32, device="cuda")]
    nxt = torch.empty(1, dtype=torch.int32, device="cuda")
    for tok, ok in ((cfg.vocab + 100, False), (11, True)):
        t = torch.tensor([tok], dtype=torch.int32, device="cuda")
        ws = ctx.decode_workspace(dm.crf, ad.crf, [20], pts, t)
        ctx.decode_step(dm.crf, ad.crf, pool, [20], pts, t, nxt, ws)
        if ok:
            ctx.check()
            assert 0 <= int(nxt.item()) < cfg.vocab
        else:
            with pytest.raises(crf.CrfError) as ei:
                ctx.check()
            assert ei.value.status == crf.abi.EINVAL


def test_debug_build_checks_page_ids_on_the_device():
    _need_gpu()
    from paper_2609_30884_gb300 import build
    build.build(debug=True)
    env = dict(os.environ, CRF_LIB_VARIANT="debug", CRF_DEBUG_DEVICE_CHECKS_ONLY="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "tests", "debug_bounds_child.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    assert "debug bounds ok" in r.stdout
