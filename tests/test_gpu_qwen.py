"""GPU parity at the Qwen2.5-shaped sizes.

* 1.5B shape, 4096-token prefix, window [20, 22): every K/V slot, both refreshed checkpoints,
  the last row carried through layers 22..27 and the first-step KL between the recovered and
  the reused state, all against the oracle run on the same inputs. With the specified adapter
  step the deep layers are dominated by the adapter (attention near one-hot, activations ~100),
  so each quantity is held to 1e-2 (1e-3 for KL) plus twice the amount the fp32 oracle itself
  moves when its steps run as a bf16 tensor pipeline (the paper's own execution); a variant with
  a 10x smaller step is held to the plain 1e-2 / 1e-3 bars.
* 1.5B shape, 16384-token prefix, the complete affected suffix [26, 28) (the window ends at the last
  layer, so the final row comes straight out of it): every K/V slot, both refreshed checkpoints,
  the final row and the first-step KL over the full 151936-token vocabulary, with the 10x smaller
  adapter step and the plain bars (the specified step's conditioning is covered at 4K above).
* 7B shape, 16384-token prefix, the launch the benchmark times (one window layer): K/V of sampled
  positions (a single-row computation for the oracle) and the layer output of sampled rows (the
  oracle projects K/V for all positions, then attends only for the sampled rows); every slot the
  request does not own stays bit-identical.
"""
from dataclasses import replace

import numpy as np
import pytest
import torch

import synth
from tests.harness import DeviceAdapter, DeviceModel, make_pool, pages_needed, split_page_tables
from oracle import build as obuild, cache as C, decoder as Dec, fidelity
from tests.gpu_util import (KL_ABS, REL_KVH, bf16_round, free_slots, oracle_adapter, oracle_model,
                            oracle_pool, rel_frob, request_kv, snapshot, bf16_execution_recover,
                            to_np, untouched_mask)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30884_gb300 as crf
    return crf.Context(0)


def _qwen15b_window(ctx, step_std, workload="1.5b-4k", window=None, bf16_reference=True):
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
    spool = oracle_pool(pool)
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
    _, h_last = C.recover(om, oa, opool, oreq, s, e, restart=restart)
    if bf16_reference:
        sreq = C.RequestCache(np.zeros(n, np.int64), pt.cpu().numpy())
        sk, sv, sh, s_final = bf16_execution_recover(om, oa, spool, sreq, s, e, restart)

    # bar: 1e-2 of the fp32 oracle plus twice what bf16 execution moves the same quantity
    report = []
    for l in range(s, e):
        for j, (name, gp, op) in enumerate((("k", pool.k_pages, opool.k), ("v", pool.v_pages, opool.v))):
            want = request_kv(torch.from_numpy(op[l]), pt, n)
            cond = rel_frob((sk, sv)[j][l], want) if bf16_reference else 0.0
            report.append((f"{name}{l}", rel_frob(request_kv(gp[l], pt, n), want), REL_KVH + 2 * cond))
        cond = rel_frob(sh[l], oreq.hidden[l]) if bf16_reference else 0.0
        report.append((f"h{l}", rel_frob(to_np(h_out[l - s]), oreq.hidden[l]), REL_KVH + 2 * cond))
    cond = rel_frob(s_final, h_last) if bf16_reference else 0.0
    report.append(("final", rel_frob(to_np(fin), h_last), REL_KVH + 2 * cond))
    report.append(("final_reuse", rel_frob(to_np(fin_reuse), h_reuse), REL_KVH))
    z_reuse = C.logits(om, h_reuse)
    want_kl = fidelity.kl(C.logits(om, h_last), z_reuse)[0]
    s_kl = fidelity.kl(C.logits(om, s_final), z_reuse)[0] if bf16_reference else want_kl
    report.append(("kl", abs(float(out_kl.item()) - want_kl), KL_ABS + 2 * abs(s_kl - want_kl)))
    print("step", step_std, "(name, err, bar):", [(a, round(b, 5), round(c, 5)) for a, b, c in report])
    for name, err, tol in report:
        assert err <= tol, (name, err, tol)
    free = untouched_mask(P, [(pt, n)])
    for l in range(cfg.n_layers):
        if s <= l < e:
            assert torch.equal(free_slots(pool.k_pages[l], free), free_slots(bk[l], free))
        else:
            assert torch.equal(pool.k_pages[l], bk[l]) and torch.equal(pool.v_pages[l], bv[l])
    return report


def test_qwen15b_4k_window_and_tail(ctx):
    """The 1.5B-shape 4K workload as specified (version step 0.005 (1 + layer))."""
    _qwen15b_window(ctx, synth.LORA_QWEN.step_std)


def test_qwen15b_4k_well_conditioned_plain_bars(ctx):
    """Same shapes and window with a 10x smaller adapter step: the plain 1e-2 / 1e-3 bars hold."""
    report = _qwen15b_window(ctx, synth.LORA_QWEN.step_std / 10)
    for name, err, _ in report:
        assert err <= (KL_ABS if name == "kl" else REL_KVH), (name, err)


def test_qwen15b_16k_suffix_well_conditioned(ctx):
    """Config of the 16K sweep, the complete affected suffix [26, 28): plain 1e-2 / 1e-3 bars."""
    report = _qwen15b_window(ctx, synth.LORA_QWEN.step_std / 10, workload="1.5b-16k", window=(26, 28),
                             bf16_reference=False)
    for name, err, tol in report:
        assert tol in (REL_KVH, KL_ABS), (name, tol)


def test_qwen7b_16k_window_layer_sampled(ctx):
    import paper_2609_30884_gb300 as crf
    wl = synth.workload("7b-16k-w1")
    cfg, lc = wl.model, wl.lora
    n = wl.n_tokens[0]
    s, e = wl.windows[0]
    dm = DeviceModel(cfg, layers=[s], with_head=False)
    cur = DeviceAdapter(cfg, lc, 1, layers=[s])
    P = pages_needed(n) + 3
    pool = make_pool(cfg, P, fill="random", seed=11)
    pt = split_page_tables([n], P, seed=5)[0]
    h_in = synth.hidden_state(cfg, n, "restart", s - 1, device="cuda")
    h_out = [torch.empty(n, cfg.hidden, dtype=torch.bfloat16, device="cuda")]
    bk, bv = snapshot(pool)
    req = crf.Request(pt, s, e, hidden_in=h_in, hidden_out=h_out)
    ws = ctx.workspace(dm.crf, cur.crf, [req])
    ctx.recompute_window(dm.crf, cur.crf, pool, [req], ws)
    ctx.check()

    P_l = oracle_model(dm).layers[s]
    A_l = oracle_adapter(cur).layers[s]
    dims = Dec.Dims(cfg.hidden, cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim, cfg.ffn, cfg.rms_eps,
                    cfg.rope_theta)
    x = to_np(h_in)
    # K/V of every position (needed by attention), computed by the oracle
    q_all, k_all, v_all = Dec.qkv(x, P_l, A_l, dims, np.arange(n))
    rows = np.array([0, 1, 15, 16, 127, 128, 4095, 8191, 12288, 16000, n - 1])
    got_k = request_kv(pool.k_pages[s], pt, n)[rows]
    got_v = request_kv(pool.v_pages[s], pt, n)[rows]
    assert rel_frob(got_k, k_all[rows]) <= REL_KVH
    assert rel_frob(got_v, v_all[rows]) <= REL_KVH
    full_k = request_kv(pool.k_pages[s], pt, n)
    assert rel_frob(full_k, k_all) <= REL_KVH          # every position's K
    # layer output of sampled rows: attention over all cached positions <= row
    got_h = to_np(h_out[0])[rows]
    want_h, alt_h = [], []
    kb, vb = bf16_round(k_all), bf16_round(v_all)
    for t in rows:
        o = Dec.single_query_attention(q_all[t], k_all[:t + 1], v_all[:t + 1])
        want_h.append(Dec.post_attention(x[t:t + 1], o[None], P_l, A_l, dims)[0])
        ob = Dec.single_query_attention(q_all[t], kb[:t + 1], vb[:t + 1])
        alt_h.append(Dec.post_attention(x[t:t + 1], ob[None], P_l, A_l, dims)[0])
    want_h = np.stack(want_h)
    sens = rel_frob(np.stack(alt_h), want_h)   # cache-format sensitivity on the sampled rows
    err = rel_frob(got_h, want_h)
    print("7B layer", s, "sampled rows: h err", err, "cache sensitivity", sens)
    assert err <= REL_KVH + 2 * sens
    free = untouched_mask(P, [(pt, n)])
    for l in range(cfg.n_layers):
        if l == s:
            assert torch.equal(free_slots(pool.k_pages[l], free), free_slots(bk[l], free))
            assert torch.equal(free_slots(pool.v_pages[l], free), free_slots(bv[l], free))
        else:
            assert torch.equal(pool.k_pages[l], bk[l])


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
