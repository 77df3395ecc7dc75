"""Offline tail-influence sweep on the device against the oracle (Sections 3.1-3.2, Eq. 2-5).

A stale cache built under adapter version 0 and the current adapter version 3 (tiny decoder, every
layer adapted): the device's N + 1 hybrid first-step distributions z^(b), their KL to the fresh
model, the tail influence T_b and the fresh margin are compared with the oracle's, and both
certificates (KL <= T_b^2 / 4; T_b < gamma*/2 keeps the top-1 token) must hold on device outputs.
"""
import numpy as np
import pytest
import torch

import synth
from tests.harness import DeviceAdapter, DeviceModel, make_pool, pages_needed, split_page_tables
from oracle import cache as C, fidelity
from tests.gpu_util import KL_ABS, oracle_adapter, oracle_model, to_np

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("n", [300, 64])
def test_tail_influence_sweep_matches_oracle(n):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30884_gb300 as crf
    from paper_2609_30884_gb300 import tail
    cfg, lc = synth.TINY, synth.LORA_TINY
    N = cfg.n_layers
    dm = DeviceModel(cfg)
    old, cur = DeviceAdapter(cfg, lc, 0), DeviceAdapter(cfg, lc, 3)
    P = pages_needed(n) + 3
    pt = split_page_tables([n], P, seed=2)[0]
    tokens = synth.token_ids(cfg, n, device="cuda")
    ctx = crf.Context(0)
    stale = make_pool(cfg, P)
    fresh_pool = make_pool(cfg, P)
    H = [torch.empty(n, cfg.hidden, dtype=torch.bfloat16, device="cuda") for _ in range(N)]
    for ad, pool, hid in ((old, stale, None), (cur, fresh_pool, H)):
        req = crf.Request(pt, 0, N, n_tokens=n, tokens=tokens, hidden_out=hid)
        ctx.recompute_window(dm.crf, ad.crf, pool, [req], ctx.workspace(dm.crf, ad.crf, [req]))
    res = tail.sweep(ctx, dm.crf, cur.crf, stale, pt, n, tokens, H, cfg.vocab)

    om, oa_old, oa_cur = oracle_model(dm), oracle_adapter(old), oracle_adapter(cur)
    tok = to_np(tokens).astype(np.int64)
    opool = C.PagedPool(N, P, cfg.n_kv_heads, cfg.head_dim)
    C.prefill(om, oa_old, opool, C.RequestCache(tok, pt.cpu().numpy()))
    freq = C.RequestCache(tok, pt.cpu().numpy())
    C.prefill(om, oa_cur, C.PagedPool(N, P, cfg.n_kv_heads, cfg.head_dim), freq)
    oreq = C.RequestCache(tok, pt.cpu().numpy())
    z = []
    for b in range(N + 1):
        start = C.embed(om, tok)[-1] if b == 0 else freq.hidden[b - 1][-1]
        z.append(C.logits(om, C.tail_decode(om, oa_cur, opool, oreq, b, start)))
    z = np.stack(z).reshape(N + 1, -1)
    want_kl = np.array([fidelity.kl(z[N][None], z[b][None])[0] for b in range(N + 1)])
    want_t = fidelity.tail_influence(list(z))
    np.testing.assert_allclose(res.kl, want_kl, atol=KL_ABS, rtol=0)
    np.testing.assert_allclose(res.tail, want_t, rtol=2e-2, atol=2e-2)
    assert abs(res.margin - float(fidelity.margin(z[N]))) <= 2e-2
    assert res.kl[N] == 0.0 and res.tail[N] == 0.0
    assert res.kl_certificate_holds.all() and res.top1_certificate_holds.all()
    assert np.all(np.diff(res.tail) <= 1e-12)   # T_b is a non-increasing envelope
    assert res.kl[0] > 5 * KL_ABS                  # the stale cache matters in this setting
