"""Pins of the oracle's cache semantics: paging, window restart, reuse identities, hybrid logits."""
import numpy as np
import pytest

import synth
from oracle import build, cache as C, decoder as D, fidelity

CFG = synth.TINY
LCFG = synth.LORA_TINY


@pytest.fixture(scope="module")
def tiny():
    model = build.model(CFG)
    v0 = build.adapter(CFG, LCFG, 0)
    v1 = build.adapter(CFG, LCFG, 1)
    return model, v0, v1


def _req(n=80, seed=1):
    pages = (n + 15) // 16
    pt = synth.page_permutation(pages + 3, seed).numpy()[:pages]
    return C.RequestCache(synth.token_ids(CFG, n).numpy(), pt)


def _pool(num_pages):
    return C.PagedPool(CFG.n_layers, num_pages, CFG.n_kv_heads, CFG.head_dim)


def test_paging_slots_exact():
    pt = np.array([5, 2, 7])
    pages, off = C.PagedPool.slots(pt, 40)
    assert pages.tolist() == [5] * 16 + [2] * 16 + [7] * 8
    assert off.tolist() == list(range(16)) * 2 + list(range(8))


def test_write_touches_only_request_slots():
    pool = _pool(10)
    pt = np.array([4, 1, 8])
    k = np.arange(35 * 2 * 64, dtype=np.float32).reshape(35, 2, 64) + 1
    pool.write(1, pt, k, -k)
    kk, vv = pool.read(1, pt, 35)
    np.testing.assert_array_equal(kk, k)
    np.testing.assert_array_equal(vv, -k)
    untouched = [p for p in range(10) if p not in (4, 1, 8)]
    assert not pool.k[1][untouched].any() and not pool.k[0].any() and not pool.k[2].any()
    assert not pool.k[1][8, :, 3:].any()          # slots past the prefix end


def test_prefill_equals_hand_unrolled_layer_loop(tiny):
    """Fresh prefill against the decoder layers composed by hand from the embedding (Eq. S1:
    H_l = F_l(H_{l-1}), C_l = G_l(H_{l-1}), H_{-1} = E[tokens]), with each layer's K/V read back
    from page page_table[t // 16], slot t % 16 by direct indexing of the pool arrays."""
    model, v0, _ = tiny
    req = _req(n=83)
    pool = _pool(16)
    C.prefill(model, v0, pool, req)
    x = model.embed[req.tokens].astype(np.float32)
    np.testing.assert_array_equal(req.hidden[-1], x)
    t = np.arange(req.n)
    for l in range(CFG.n_layers):
        x, k, v = D.decoder_layer(x, model.layers[l], v0.layers[l], model.dims)
        np.testing.assert_array_equal(pool.k[l][req.page_table[t // 16], :, t % 16, :], k)
        np.testing.assert_array_equal(pool.v[l][req.page_table[t // 16], :, t % 16, :], v)
        np.testing.assert_array_equal(req.hidden[l], x)


def test_split_windows_compose_to_prefill(tiny):
    """Two windows [0, 2) and [2, N), the second restarting from the first's H_1, leave the same
    cache and checkpoints as one fresh prefill: restart from a retained boundary state (Section 4.2)."""
    model, v0, _ = tiny
    r1, r2 = _req(), _req()
    p1, p2 = _pool(16), _pool(16)
    C.prefill(model, v0, p1, r1)
    C.run_window(model, v0, p2, r2, 0, 2)
    x = C.run_window(model, v0, p2, r2, 2, CFG.n_layers)
    for l in range(CFG.n_layers):
        np.testing.assert_array_equal(p1.k[l], p2.k[l])
        np.testing.assert_array_equal(p1.v[l], p2.v[l])
        np.testing.assert_array_equal(r1.hidden[l], r2.hidden[l])
    np.testing.assert_array_equal(x, r1.hidden[CFG.n_layers - 1])


def test_identical_adapter_reproduces_stale_cache(tiny):
    model, v0, _ = tiny
    req = _req()
    pool = _pool(16)
    C.prefill(model, v0, pool, req)
    before = pool.copy()
    h_before = {l: a.copy() for l, a in req.hidden.items()}
    C.run_window(model, v0, pool, req, 1, 3)
    for l in range(CFG.n_layers):
        np.testing.assert_array_equal(pool.k[l], before.k[l])
        np.testing.assert_array_equal(pool.v[l], before.v[l])
    for l in range(1, 3):
        np.testing.assert_array_equal(req.hidden[l], h_before[l])


def test_window_overwrites_only_its_layers(tiny):
    model, v0, v1 = tiny
    req = _req()
    pool = _pool(16)
    C.prefill(model, v0, pool, req)
    before = pool.copy()
    C.run_window(model, v1, pool, req, 2, 3)
    for l in (0, 1, 3):
        np.testing.assert_array_equal(pool.k[l], before.k[l])
    assert not np.array_equal(pool.k[2], before.k[2])


def test_query_only_update_one_layer_window_is_stale_reuse(tiny):
    """Eq. S4: after a query-only update at layer s, executing [s, s+1) replaces no K/V."""
    model, v0, _ = tiny
    s = 1
    vq = C.Adapter([D.LayerAdapter(dict(a.AB), a.scale) for a in v0.layers])
    A, B = vq.layers[s].AB["q"]
    vq.layers[s].AB["q"] = (A + 0.05, B - 0.05)
    req = _req()
    pool = _pool(16)
    C.prefill(model, v0, pool, req)
    before = pool.copy()
    h_old = req.hidden[s].copy()
    C.run_window(model, vq, pool, req, s, s + 1)
    for l in range(CFG.n_layers):
        np.testing.assert_array_equal(pool.k[l], before.k[l])
        np.testing.assert_array_equal(pool.v[l], before.v[l])
    assert not np.allclose(req.hidden[s], h_old)       # the hidden state did change


def test_key_update_one_layer_window_changes_that_layer(tiny):
    model, v0, _ = tiny
    s = 1
    vk = C.Adapter([D.LayerAdapter(dict(a.AB), a.scale) for a in v0.layers])
    A, B = vk.layers[s].AB["k"]
    vk.layers[s].AB["k"] = (A + 0.05, B - 0.05)
    req, pool = _req(), _pool(16)
    C.prefill(model, v0, pool, req)
    before = pool.copy()
    C.run_window(model, vk, pool, req, s, s + 1)
    assert not np.array_equal(pool.k[s], before.k[s])
    np.testing.assert_array_equal(pool.v[s], before.v[s])


def test_tail_decode_over_fresh_cache_gives_fresh_logits(tiny):
    """z^(b) with a cache that is already fresh at every layer equals z* for any boundary."""
    model, _, v1 = tiny
    req, pool = _req(), _pool(16)
    x = C.prefill(model, v1, pool, req)
    z_star = C.logits(model, x[-1])
    for e in range(CFG.n_layers + 1):
        h_prev = req.hidden[e - 1][-1]
        h = C.tail_decode(model, v1, pool, req, e, h_prev)
        np.testing.assert_allclose(C.logits(model, h), z_star, rtol=1e-4, atol=1e-4)


def test_full_window_recovery_has_zero_kl(tiny):
    """Exact recovery (window [0, N)) reproduces fresh logits: zero KL, top-1 agreement."""
    model, v0, v1 = tiny
    req_f, pool_f = _req(), _pool(16)
    x = C.prefill(model, v1, pool_f, req_f)
    z_star = C.logits(model, x[-1])
    req, pool = _req(), _pool(16)
    C.prefill(model, v0, pool, req)
    _, h = C.recover(model, v1, pool, req, 0, CFG.n_layers)
    z = C.logits(model, h)
    assert fidelity.kl(z_star, z)[0] == pytest.approx(0.0, abs=1e-12)
    # stale reuse (empty window) differs
    req2, pool2 = _req(), _pool(16)
    C.prefill(model, v0, pool2, req2)
    _, h_stale = C.recover(model, v1, pool2, req2, 2, 2)
    assert fidelity.kl(z_star, C.logits(model, h_stale))[0] > 1e-6


def test_recovery_with_restart_state_argument(tiny):
    model, v0, v1 = tiny
    req, pool = _req(), _pool(16)
    C.prefill(model, v0, pool, req)
    h1 = req.hidden[1].copy()
    req2, pool2 = _req(), pool.copy()
    x_a = C.run_window(model, v1, pool, req, 2, 4)
    x_b = C.run_window(model, v1, pool2, req2, 2, 4, restart=h1)
    np.testing.assert_array_equal(x_a, x_b)


def test_logits_match_library_final_norm_and_head(tiny):
    """z = W_lm (rmsnorm(h) * g_f): against torch's rms_norm and linear in float64."""
    import torch
    import torch.nn.functional as F
    model, _, _ = tiny
    rng = np.random.default_rng(11)
    h = rng.standard_normal((3, CFG.hidden)) * 2.0
    z = C.logits(model, h, np.float64)
    t = lambda a: torch.tensor(np.asarray(a, np.float64))
    want = F.linear(F.rms_norm(t(h), (CFG.hidden,), t(model.final_norm), CFG.rms_eps),
                    t(model.lm_head)).numpy()
    np.testing.assert_allclose(z, want, rtol=1e-12, atol=1e-12)
    # a single row gives its row of the batch (up to the BLAS blocking of a 1-row product)
    np.testing.assert_allclose(C.logits(model, h[1], np.float64)[0], z[1], rtol=1e-12, atol=1e-13)


def test_embed_matches_library_lookup(tiny):
    """H_{-1} = E[tokens]: against torch's embedding lookup, repeated ids included."""
    import torch
    import torch.nn.functional as F
    model, _, _ = tiny
    tokens = np.array([0, CFG.vocab - 1, 5, 5, 17])
    got = C.embed(model, tokens, np.float64)
    want = F.embedding(torch.tensor(tokens), torch.tensor(np.asarray(model.embed, np.float64))).numpy()
    np.testing.assert_array_equal(got, want)
