"""The Python binding marshals the caller's tensors into the C structs of include/crf.h: pointer
tables, module order, sizes and flags (CPU tensors stand in for device ones; no call is made)."""
import torch

import paper_2609_30884_gb300 as crf

DIMS = dict(n_layers=2, hidden=64, n_q_heads=4, n_kv_heads=2, head_dim=16, ffn=96, vocab=50,
            rms_eps=1e-6, rope_theta=1e4, qkv_bias=True)


def _addr(p):
    return p if isinstance(p, int) or p is None else p.value


def test_model_pointer_tables_follow_module_order():
    layers = []
    for l in range(2):
        w = {f"W_{m}": torch.zeros(4 + j) for j, m in enumerate(crf.MODULES)}
        w.update({f"bias_{m}": torch.zeros(2) for m in ("q", "k", "v")}, ln1=torch.zeros(3), ln2=torch.zeros(3))
        layers.append(w)
    embed, fn, head = torch.zeros(5), torch.zeros(6), torch.zeros(7)
    m = crf.Model(DIMS, layers, embed, fn, head)
    d = m.c.dims
    assert (d.n_layers, d.hidden, d.n_q_heads, d.n_kv_heads, d.head_dim, d.ffn, d.vocab, d.qkv_bias) == \
        (2, 64, 4, 2, 16, 96, 50, 1)
    for l in range(2):
        lw = m.c.layers[l]
        for j, name in enumerate(crf.MODULES):
            assert _addr(lw.W[j]) == layers[l][f"W_{name}"].data_ptr()
        for j, name in enumerate(("q", "k", "v")):
            assert _addr(lw.bias[j]) == layers[l][f"bias_{name}"].data_ptr()
        assert _addr(lw.ln1) == layers[l]["ln1"].data_ptr() and _addr(lw.ln2) == layers[l]["ln2"].data_ptr()
    assert (_addr(m.c.embed), _addr(m.c.final_norm), _addr(m.c.lm_head)) == \
        (embed.data_ptr(), fn.data_ptr(), head.data_ptr())


def test_model_without_bias_or_head_passes_nulls():
    layers = [{f"W_{m}": torch.zeros(2) for m in crf.MODULES} | {"ln1": torch.zeros(1), "ln2": torch.zeros(1)}, None]
    m = crf.Model(dict(DIMS, qkv_bias=False), layers)
    assert m.c.dims.qkv_bias == 0
    assert all(_addr(m.c.layers[0].bias[j]) is None for j in range(3))
    assert _addr(m.c.layers[1].W[0]) is None          # a layer the caller left out
    assert _addr(m.c.embed) is None and _addr(m.c.lm_head) is None


def test_adapter_tables_are_layer_major_with_module_mask():
    A = {(l, m): torch.zeros(3) for l in range(2) for m in ("v", "down")}
    B = {(l, m): torch.zeros(3) for l in range(2) for m in ("v", "down")}
    ad = crf.Adapter(8, 16.0, ("v", "down"), [{m: (A[l, m], B[l, m]) for m in ("v", "down")} for l in range(2)])
    assert (ad.c.dims.rank, ad.c.dims.alpha) == (8, 16.0)
    assert ad.c.dims.module_mask == (1 << 2) | (1 << 6)
    for l in range(2):
        for j, name in enumerate(crf.MODULES):
            a, b = _addr(ad.c.A[l * 7 + j]), _addr(ad.c.B[l * 7 + j])
            if name in ("v", "down"):
                assert a == A[l, name].data_ptr() and b == B[l, name].data_ptr()
            else:
                assert a is None and b is None


def test_request_and_pool_marshalling():
    pt = torch.arange(3, dtype=torch.int32)
    toks = torch.zeros(40, dtype=torch.int32)
    outs = [torch.zeros(40, 8) for _ in range(2)]
    fin = torch.zeros(8)
    r = crf.Request(pt, 0, 2, tokens=toks, hidden_out=outs, final_hidden_out=fin)
    c = r.c
    assert (c.n_tokens, c.s, c.e) == (40, 0, 2)
    assert _addr(c.page_table) == pt.data_ptr() and _addr(c.tokens) == toks.data_ptr()
    assert _addr(c.hidden_in) is None and _addr(c.final_hidden_out) == fin.data_ptr()
    assert [c.hidden_out[i] for i in range(2)] == [o.data_ptr() for o in outs]
    h_in = torch.zeros(33, 8)
    r2 = crf.Request(pt, 1, 1, hidden_in=h_in)        # n_tokens from hidden_in; empty window
    assert (r2.c.n_tokens, r2.c.s, r2.c.e) == (33, 1, 1) and not r2.c.hidden_out
    ks = [torch.zeros(5, 2, 16, 16) for _ in range(2)]
    vs = [torch.zeros(5, 2, 16, 16) for _ in range(2)]
    pool = crf.KVPool(ks, vs)
    assert pool.c.num_pages == 5
    assert [pool.c.k_pages[i] for i in range(2)] == [k.data_ptr() for k in ks]
    assert [pool.c.v_pages[i] for i in range(2)] == [v.data_ptr() for v in vs]


def test_decode_rows_point_at_each_token():
    toks = torch.tensor([7, 8, 9], dtype=torch.int32)
    pts = [torch.zeros(2, dtype=torch.int32) for _ in range(3)]
    rows = crf.Context._decode_rows([20, 31, 5], pts, toks)
    assert [rows[i].pos for i in range(3)] == [20, 31, 5]
    assert [rows[i].page_table for i in range(3)] == [p.data_ptr() for p in pts]
    assert [rows[i].token for i in range(3)] == [toks.data_ptr() + 4 * i for i in range(3)]
