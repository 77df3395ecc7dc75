"""GPU parity at the Qwen2.5 1.5B shape (the 7B benchmarked step is test_gpu_bench_parity.py).

* 4096-token prefix, window [20, 22) with the specified adapter step 0.005 (1 + layer): every
  K/V slot and every row of both refreshed checkpoints, each window layer against the oracle's
  layer run on the GPU's own input for that layer; the last row carried through layers 22..27
  against the oracle's tail decode of the GPU's window output over the same pages; the
  first-step KL against the oracle's KL of the oracle's own rows. The deep layers of this adapter
  are adapter-dominated (attention near one-hot, activations ~100), and a layer's own bar is
  1e-2 or 1.25x the distance its oracle layer moves when it stores its intermediates in bf16
  where the path does, whichever is larger.
* The same shapes with a 10x smaller adapter step, chained end to end from the restart state
  (pages, checkpoints, final row, KL) under the plain 1e-2 / 1e-3 bars.
* 16384-token prefix, the complete affected suffix [26, 28) with the 10x smaller step, chained
  end to end under the plain bars, over the full 151936-token vocabulary.
"""
from dataclasses import replace

import numpy as np
import pytest
import torch

import synth
from tests.harness import DeviceAdapter, DeviceModel, make_pool, pages_needed, split_page_tables
from oracle import cache as C, fidelity
from tests.gpu_util import (KL_ABS, REL_KVH, free_slots, local_layer_report, oracle_adapter,
                            oracle_model, oracle_pool, rel_frob, request_kv, snapshot, to_np,
                            untouched_mask)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30884_gb300 as crf
    return crf.Context(0)


def _qwen15b_window(ctx, step_std, workload="1.5b-4k", window=None, local=False):
    """Run window [s, e) + tail + KL against direct reuse on the GPU; return [(name, err, bar)].

    local=False: chained from the restart state against the oracle's own window (plain bars).
    local=True: each window layer on the GPU's own input, the tail from the GPU's window output."""
    import paper_2609_30884_gb300 as crf
    wl = synth.workload(workload)
    cfg = wl.model
    lc = replace(wl.lora, step_std=step_std)
    n = wl.n_tokens[0]
    s, e = window if window is not None else wl.windows[0]
    dm = DeviceModel(cfg, layers=range(s, cfg.n_layers))
    cur = DeviceAdapter(cfg, lc, 1, layers=range(s, cfg.n_layers))
    P = pages_needed(n) + 5
    pool = make_pool(cfg, P, fill="random", seed=7)
    pt = split_page_tables([n], P, seed=3)[0]
    h_in = synth.hidden_state(cfg, n, "restart", s - 1, device="cuda")
    h_out = [torch.empty(n, cfg.hidden, dtype=torch.bfloat16, device="cuda") for _ in range(e - s)]
    fin = torch.empty(cfg.hidden, dtype=torch.bfloat16, device="cuda")
    fin_reuse = torch.empty(cfg.hidden, dtype=torch.bfloat16, device="cuda")
    bk, bv = snapshot(pool)
    opool = oracle_pool(pool)
    # direct reuse first (reads the historical pages of layers s..N-1), then the window
    reuse = crf.Request(pt, s, s, n_tokens=n, hidden_in=h_in, final_hidden_out=fin_reuse)
    ctx.recompute_window(dm.crf, cur.crf, pool, [reuse], ctx.workspace(dm.crf, cur.crf, [reuse]))
    req = crf.Request(pt, s, e, hidden_in=h_in, hidden_out=h_out, final_hidden_out=fin)
    ctx.recompute_window(dm.crf, cur.crf, pool, [req], ctx.workspace(dm.crf, cur.crf, [req]))
    out_kl = torch.empty(1, dtype=torch.float32, device="cuda")
    ctx.kl(dm.crf, fin[None], fin_reuse[None], out_kl, cfg.vocab,
           ctx.kl_workspace(1, cfg.vocab, cfg.hidden))
    ctx.check()

    om, oa = oracle_model(dm), oracle_adapter(cur)
    oreq = C.RequestCache(np.zeros(n, np.int64), pt.cpu().numpy())
    restart = to_np(h_in)
    h_reuse = C.tail_decode(om, oa, opool, oreq, s, restart[-1])
    report = []
    if local:
        x_in = restart
        for l in range(s, e):
            got_h = to_np(h_out[l - s])
            report += [(a, b, c) for a, b, c, _ in local_layer_report(
                x_in, om.layers[l], oa.layers[l], om.dims, got_h, request_kv(pool.k_pages[l], pt, n),
                request_kv(pool.v_pages[l], pt, n), str(l))]
            x_in = got_h
        # the oracle's tail of the GPU's window output over the same (historical) pages
        h_last = C.tail_decode(om, oa, opool, oreq, e, x_in[-1])
    else:
        _, h_last = C.recover(om, oa, opool, oreq, s, e, restart=restart)
        for l in range(s, e):
            for name, gp, op in (("k", pool.k_pages, opool.k), ("v", pool.v_pages, opool.v)):
                want = request_kv(torch.from_numpy(op[l]), pt, n)
                report.append((f"{name}{l}", rel_frob(request_kv(gp[l], pt, n), want), REL_KVH))
            report.append((f"h{l}", rel_frob(to_np(h_out[l - s]), oreq.hidden[l]), REL_KVH))
    report.append(("final", rel_frob(to_np(fin), h_last), REL_KVH))
    report.append(("final_reuse", rel_frob(to_np(fin_reuse), h_reuse), REL_KVH))
    want_kl = fidelity.kl(C.logits(om, h_last), C.logits(om, h_reuse))[0]
    report.append(("kl", abs(float(out_kl.item()) - want_kl), KL_ABS))
    print("step", step_std, "local" if local else "chained", "(name, err, bar):",
          [(a, round(b, 5), round(c, 5)) for a, b, c in report])
    for name, err, tol in report:
        assert err <= tol, (name, err, tol)
    free = untouched_mask(P, [(pt, n)])
    for l in range(cfg.n_layers):
        if s <= l < e:
            assert torch.equal(free_slots(pool.k_pages[l], free), free_slots(bk[l], free))
            assert torch.equal(free_slots(pool.v_pages[l], free), free_slots(bv[l], free))
        else:
            assert torch.equal(pool.k_pages[l], bk[l]) and torch.equal(pool.v_pages[l], bv[l])
    return report


def test_qwen15b_4k_window_and_tail(ctx):
    """The 1.5B-shape 4K workload as specified (version step 0.005 (1 + layer)), layer by layer."""
    _qwen15b_window(ctx, synth.LORA_QWEN.step_std, local=True)


def test_qwen15b_4k_well_conditioned_plain_bars(ctx):
    """Same shapes and window with a 10x smaller adapter step, chained: the plain bars hold."""
    report = _qwen15b_window(ctx, synth.LORA_QWEN.step_std / 10)
    assert all(tol in (REL_KVH, KL_ABS) for _, _, tol in report)


def test_qwen15b_16k_suffix_well_conditioned(ctx):
    """Config of the 16K sweep, the complete affected suffix [26, 28), chained: plain bars."""
    report = _qwen15b_window(ctx, synth.LORA_QWEN.step_std / 10, workload="1.5b-16k", window=(26, 28))
    assert all(tol in (REL_KVH, KL_ABS) for _, _, tol in report)


def test_misaligned_bias_rejected(ctx):
    """The QKV epilogue reads biases as 16-byte vectors: a bias pointer off that boundary is
    refused on the host (CRF_EINVAL) before anything is launched, and the pages stay untouched."""
    import paper_2609_30884_gb300 as crf
    cfg = replace(synth.QWEN15B, name="qwen2.5-1.5b-shape-2l", n_layers=2)
    lc = synth.LORA_QWEN
    dm = DeviceModel(cfg, with_head=False)
    cur = DeviceAdapter(cfg, lc, 1)
    n = 256
    P = pages_needed(n)
    pool = make_pool(cfg, P)
    pt = split_page_tables([n], P, seed=3)[0]
    h = synth.hidden_state(cfg, n, device="cuda")
    layers = [dict(w) for w in dm.layers]
    b = layers[1]["bias_k"]
    padded = torch.empty(b.numel() + 1, dtype=b.dtype, device=b.device)
    padded[1:].copy_(b)
    layers[1]["bias_k"] = padded[1:]  # starts 2 bytes past a 16-byte boundary
    bad = crf.Model(dm.crf.dims, layers)
    req = crf.Request(pt, 1, 2, hidden_in=h)
    ws = ctx.workspace(bad, cur.crf, [req])
    bk = [k.clone() for k in pool.k_pages]
    with pytest.raises(crf.CrfError) as ei:
        ctx.recompute_window(bad, cur.crf, pool, [req], ws)
    assert ei.value.status == crf.abi.EINVAL
    torch.cuda.synchronize()
    assert all(torch.equal(a, c) for a, c in zip(pool.k_pages, bk))
    ctx.recompute_window(dm.crf, cur.crf, pool, [req], ws)  # the aligned model still runs
    ctx.check()
