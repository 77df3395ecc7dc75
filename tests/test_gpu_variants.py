"""GPU parity for adapter rank and module variants.

The paper's ablations adapt fewer modules (a value-only adapter, Section 5.5) and its main runs use
rank 8; the hot path is specialised by rank (padded to one 16-wide K step) and module mask. Each
variant runs a window plus the first-step row and its KL against the oracle, on the tiny decoder
(head dim 64) and on a 4-layer decoder with the Qwen2.5-1.5B layer shapes (head dim 128, q/k/v
bias), with a ragged prefix; the drift of each variant is checked against the factored oracle.
"""
from dataclasses import replace

import numpy as np
import pytest
import torch

import synth
from tests.harness import DeviceAdapter, DeviceModel, make_pool, pages_needed, split_page_tables
from oracle import cache as C, drift as odrift, fidelity
from tests.gpu_util import (DRIFT_REL, KL_ABS, REL_KVH, oracle_adapter, oracle_model, oracle_pool,
                            rel_frob, request_kv, snapshot, to_np, untouched_mask, free_slots)

pytestmark = pytest.mark.gpu

VARIANTS = [
    (4, synth.MODULES),
    (8, ("v",)),
    (8, ("q", "v")),
    (16, ("o",)),
    (16, ("gate", "down")),
    (8, ("up",)),
]
# 4 layers with the 1.5B layer shapes; the well-conditioned adapter step keeps plain bars meaningful
SMALL128 = replace(synth.QWEN15B, name="qwen2.5-1.5b-shape-4l", n_layers=4)
SHAPES = {"tiny": (synth.TINY, 300, (1, 3)), "1.5b-4l": (SMALL128, 700, (1, 3))}


@pytest.fixture(scope="module")
def ctx():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30884_gb300 as crf
    return crf.Context(0)


@pytest.fixture(scope="module")
def models():
    return {k: DeviceModel(cfg) for k, (cfg, _, _) in SHAPES.items()}


def _lcfg(rank, modules, cfg):
    # alpha / r = 2 as in the specified configurations; a 10x smaller version step on the
    # 1.5B shapes, whose deep layers otherwise amplify bf16 rounding beyond the plain bars
    step = 0.005 if cfg is synth.TINY else 0.0005
    return synth.LoraCfg(rank, 2.0 * rank, tuple(modules), step_std=step)


@pytest.mark.parametrize("rank,modules", VARIANTS, ids=[f"r{r}-{'+'.join(m) if len(m) < 7 else 'all'}"
                                                         for r, m in VARIANTS])
@pytest.mark.parametrize("shape", list(SHAPES))
def test_variant_window_tail_kl(ctx, models, shape, rank, modules):
    import paper_2609_30884_gb300 as crf
    cfg, n, (s, e) = SHAPES[shape]
    lc = _lcfg(rank, modules, cfg)
    dm = models[shape]
    cur = DeviceAdapter(cfg, lc, 1)
    P = pages_needed(n) + 5
    pool = make_pool(cfg, P, fill="random", seed=21)
    pt = split_page_tables([n], P, seed=4)[0]
    h_in = synth.hidden_state(cfg, n, "restart", 7, device="cuda")
    h_out = [torch.empty(n, cfg.hidden, dtype=torch.bfloat16, device="cuda") for _ in range(e - s)]
    fin = torch.empty(cfg.hidden, dtype=torch.bfloat16, device="cuda")
    fin_reuse = torch.empty(cfg.hidden, dtype=torch.bfloat16, device="cuda")
    bk, bv = snapshot(pool)
    opool = oracle_pool(pool)
    reuse = crf.Request(pt, s, s, n_tokens=n, hidden_in=h_in, final_hidden_out=fin_reuse)
    ctx.recompute_window(dm.crf, cur.crf, pool, [reuse], ctx.workspace(dm.crf, cur.crf, [reuse]))
    req = crf.Request(pt, s, e, hidden_in=h_in, hidden_out=h_out, final_hidden_out=fin)
    ctx.recompute_window(dm.crf, cur.crf, pool, [req], ctx.workspace(dm.crf, cur.crf, [req]))
    out_kl = torch.empty(1, dtype=torch.float32, device="cuda")
    ctx.kl(dm.crf, fin[None], fin_reuse[None], out_kl, cfg.vocab, ctx.kl_workspace(1, cfg.vocab, cfg.hidden))
    ctx.check()

    om, oa = oracle_model(dm), oracle_adapter(cur)
    oreq = C.RequestCache(np.zeros(n, np.int64), pt.cpu().numpy())
    restart = to_np(h_in)
    h_reuse = C.tail_decode(om, oa, opool, oreq, s, restart[-1])
    _, h_last = C.recover(om, oa, opool, oreq, s, e, restart=restart)
    for l in range(s, e):
        for name, gp, op in (("k", pool.k_pages, opool.k), ("v", pool.v_pages, opool.v)):
            err = rel_frob(request_kv(gp[l], pt, n), request_kv(torch.from_numpy(op[l]), pt, n))
            assert err <= REL_KVH, (name, l, err)
        assert rel_frob(to_np(h_out[l - s]), oreq.hidden[l]) <= REL_KVH, ("h", l)
    assert rel_frob(to_np(fin), h_last) <= REL_KVH
    assert rel_frob(to_np(fin_reuse), h_reuse) <= REL_KVH
    want_kl = fidelity.kl(C.logits(om, h_last), C.logits(om, h_reuse))[0]
    assert abs(float(out_kl.item()) - want_kl) <= KL_ABS, (float(out_kl.item()), want_kl)
    # slots the request does not own and layers outside the window stay bit-identical
    free = untouched_mask(P, [(pt, n)])
    for l in range(cfg.n_layers):
        if s <= l < e:
            assert torch.equal(free_slots(pool.k_pages[l], free), free_slots(bk[l], free))
        else:
            assert torch.equal(pool.k_pages[l], bk[l]) and torch.equal(pool.v_pages[l], bv[l])


@pytest.mark.parametrize("rank,modules", VARIANTS[:3], ids=["r4-all", "r8-v", "r8-q+v"])
def test_variant_drift(ctx, rank, modules):
    cfg = SMALL128
    lc = _lcfg(rank, modules, cfg)
    cur = DeviceAdapter(cfg, lc, 2)
    anchor = DeviceAdapter(cfg, lc, 0)
    out = torch.empty(cfg.n_layers, 7, 2, dtype=torch.float32, device="cuda")
    from tests.test_gpu_kl_drift import _dims_c
    ws = ctx.drift_workspace(_dims_c(cfg), cur.crf.dims_c)
    ctx.drift(_dims_c(cfg), cur.crf, [anchor.crf] * cfg.n_layers, out, ws)
    ctx.check()
    got = to_np(out).astype(np.float64)
    oc, o0 = oracle_adapter(cur).layers, oracle_adapter(anchor).layers
    for l in range(cfg.n_layers):
        for j, m in enumerate(synth.MODULES):
            if m not in modules:
                assert got[l, j, 0] == 0 and got[l, j, 1] == 0
                continue
            A0, B0 = o0[l].AB[m]
            A1, B1 = oc[l].AB[m]
            for k, ref in enumerate((odrift.factored_sq(A0, B0, A1, B1), odrift.param_sq(A0, B0, A1, B1))):
                assert abs(got[l, j, k] - ref) <= DRIFT_REL * ref, (l, m, k, got[l, j, k], ref)
