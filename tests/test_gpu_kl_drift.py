"""GPU parity of crf_kl and crf_drift against the oracle."""
import numpy as np
import pytest
import torch

import synth
from tests.harness import DeviceAdapter, DeviceModel
from oracle import cache as C, drift as odrift, fidelity
from tests.gpu_util import DRIFT_REL, KL_ABS, oracle_adapter, oracle_model, rel_frob, to_np

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30884_gb300 as crf
    return crf.Context(0)


@pytest.mark.parametrize("rows,vocab,scale", [(1, 1024, 1.0), (3, 152064, 3.0), (4, 151936, 0.2),
                                              (2, 5, 1.0)])
def test_kl_from_logits(ctx, rows, vocab, scale):
    z_ref = synth.normal((rows, vocab), "zref", 0, scale, device="cuda")
    z_cur = z_ref + synth.normal((rows, vocab), "dz", 0, 0.3 * scale, device="cuda")
    out = torch.empty(rows, dtype=torch.float32, device="cuda")
    ws = ctx.kl_workspace(rows, vocab)
    ctx.kl(None, z_ref, z_cur, out, vocab, ws)
    ctx.check()
    want = fidelity.kl(to_np(z_ref).astype(np.float64), to_np(z_cur).astype(np.float64))
    np.testing.assert_allclose(to_np(out), want, atol=KL_ABS, rtol=0)
    np.testing.assert_allclose(to_np(out), want, rtol=1e-3, atol=1e-5)
    # KL(p || p) = 0
    ctx.kl(None, z_ref, z_ref, out, vocab, ws)
    torch.cuda.synchronize()
    assert np.all(np.abs(to_np(out)) < 1e-5)


@pytest.mark.parametrize("cfg", [synth.TINY, synth.QWEN15B], ids=["tiny", "1.5b"])
def test_kl_with_model_head(ctx, cfg):
    dm = DeviceModel(cfg, layers=[])
    om = oracle_model(dm)
    rows = 2
    h_ref = synth.hidden_state(cfg, rows, "href", std=2.0, device="cuda")
    h_cur = (h_ref.float() + synth.normal((rows, cfg.hidden), "dh", 0, 0.3, device="cuda")).bfloat16()
    out = torch.empty(rows, dtype=torch.float32, device="cuda")
    logits = torch.empty(2 * rows, cfg.vocab, dtype=torch.float32, device="cuda")
    ws = ctx.kl_workspace(rows, cfg.vocab, cfg.hidden)
    ctx.kl(dm.crf, h_ref, h_cur, out, cfg.vocab, ws, logits_out=logits)
    ctx.check()
    zr = C.logits(om, to_np(h_ref))
    zc = C.logits(om, to_np(h_cur))
    assert rel_frob(to_np(logits[:rows]), zr) < 1e-4
    assert rel_frob(to_np(logits[rows:]), zc) < 1e-4
    np.testing.assert_allclose(to_np(out), fidelity.kl(zr, zc), atol=KL_ABS, rtol=0)
    # Eq. 4 certificate on the device logits
    lg = to_np(logits).astype(np.float64)
    bound = 0.25 * np.sum((lg[rows:] - lg[:rows]) ** 2, axis=1)
    assert np.all(to_np(out) <= bound + 1e-4)


@pytest.mark.parametrize("cfg,lc", [(synth.TINY, synth.LORA_TINY), (synth.QWEN15B, synth.LORA_QWEN)],
                         ids=["tiny-r8", "1.5b-r16"])
def test_drift_matches_oracle(ctx, cfg, lc):
    n = cfg.n_layers
    cur = DeviceAdapter(cfg, lc, 3)
    anchors = {v: DeviceAdapter(cfg, lc, v) for v in (0, 1, 3)}
    # mixed-version cache: every layer has its own anchor
    which = [(0, 1, 3)[l % 3] for l in range(n)]
    out = torch.empty(n, 7, 2, dtype=torch.float32, device="cuda")
    ws = ctx.drift_workspace(_dims_c(cfg), cur.crf.dims_c)
    ctx.drift(_dims_c(cfg), cur.crf, [anchors[a].crf for a in which], out, ws)
    ctx.check()
    got = to_np(out).astype(np.float64)
    oc = oracle_adapter(cur).layers
    ref = np.zeros((n, 7, 2))
    anc_np = {v: oracle_adapter(a).layers for v, a in anchors.items()}
    for l in range(n):
        for j, m in enumerate(synth.MODULES):
            if m not in lc.modules:
                continue
            A0, B0 = anc_np[which[l]][l].AB[m]
            A1, B1 = oc[l].AB[m]
            ref[l, j, 0] = odrift.factored_sq(A0, B0, A1, B1)
            ref[l, j, 1] = odrift.param_sq(A0, B0, A1, B1)
    nz = ref > 0
    assert np.all(got[~nz] == 0)
    rel = np.abs(got[nz] - ref[nz]) / ref[nz]
    assert rel.max() <= DRIFT_REL, f"max rel drift error {rel.max():.3e}"
    # identical versions give exactly zero
    assert np.all(got[[l for l in range(n) if which[l] == 3]] == 0)


def test_drift_more_items_than_one_launch(ctx):
    """240 (layer, module) items, more than one launch pair takes: the host splits them over two
    Gram + combine launches that reuse one workspace. Every adapted entry matches the factored
    oracle (down's 688-wide input ends in a 176-column step, zero-filled past its columns); the
    unadapted v entries, poisoned with NaN first, read zero."""
    cfg = synth.replace(synth.TINY, n_layers=40)
    lc = synth.replace(synth.LORA_TINY, rank=16, modules=("q", "k", "o", "gate", "up", "down"))
    cur, anchor = DeviceAdapter(cfg, lc, 2), DeviceAdapter(cfg, lc, 0)
    out = torch.full((cfg.n_layers, 7, 2), float("nan"), dtype=torch.float32, device="cuda")
    ws = ctx.drift_workspace(_dims_c(cfg), cur.crf.dims_c)
    ctx.drift(_dims_c(cfg), cur.crf, [anchor.crf] * cfg.n_layers, out, ws)
    ctx.check()
    got = to_np(out).astype(np.float64)
    oc, oa = oracle_adapter(cur).layers, oracle_adapter(anchor).layers
    worst = 0.0
    for l in range(cfg.n_layers):
        for j, m in enumerate(synth.MODULES):
            if m not in lc.modules:
                assert got[l, j, 0] == 0.0 and got[l, j, 1] == 0.0, (l, m)
                continue
            A0, B0 = oa[l].AB[m]
            A1, B1 = oc[l].AB[m]
            for k, ref in enumerate((odrift.factored_sq(A0, B0, A1, B1), odrift.param_sq(A0, B0, A1, B1))):
                worst = max(worst, abs(got[l, j, k] - ref) / ref)
    assert worst <= DRIFT_REL, f"max rel drift error {worst:.3e}"


def _dims_c(cfg):
    from paper_2609_30884_gb300 import abi
    return abi.ModelDims(cfg.n_layers, cfg.hidden, cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim,
                         cfg.ffn, cfg.vocab, cfg.rms_eps, cfg.rope_theta, int(cfg.qkv_bias))
