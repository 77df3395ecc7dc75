"""The allocation-free KL entry point agrees with the workspace one.

crf_kl_logits_noalloc exists for callers that cannot allocate device memory
when they need the fidelity number; it keeps its scratch in a fixed device
array of the library. This file is collected last so that a run stopping at
the first failure has already run every other test.
"""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

KL_ABS = 1e-3   # the KL tolerance of the parity tests


def _kl_workspace_path(ctx, z_ref, z_cur):
    out = torch.empty(z_ref.shape[0], dtype=torch.float32, device="cuda")
    ws = ctx.kl_workspace(z_ref.shape[0], z_ref.shape[1])
    ctx.kl(None, z_ref, z_cur, out, z_ref.shape[1], ws)
    torch.cuda.synchronize()
    return out.cpu().numpy()


def test_noalloc_kl_matches_workspace_kl_twice():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_30884_gb300 import build
    build.build()
    import paper_2609_30884_gb300 as crf
    ctx = crf.Context(0)
    rows, vocab = 3, 152064
    z_ref = synth.normal((rows, vocab), "noalloc_ref", 0, 2.0, device="cuda")
    for call in range(2):       # two calls in a row share the fixed scratch
        z_cur = z_ref + synth.normal((rows, vocab), "noalloc_cur", call, 0.3 + call, device="cuda")
        want = _kl_workspace_path(ctx, z_ref, z_cur)
        out = torch.full((rows,), float("nan"), dtype=torch.float32, device="cuda")
        crf.kl_logits_noalloc(0, z_ref, z_cur, out)
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        np.testing.assert_allclose(got, want, atol=KL_ABS, rtol=0)
        assert np.all(np.isfinite(got)) and np.all(got > 0)
    too_many = torch.zeros(33, 8, dtype=torch.float32, device="cuda")
    with pytest.raises(crf.CrfError) as ei:
        crf.kl_logits_noalloc(0, too_many, too_many, torch.empty(33, device="cuda"))
    assert ei.value.status == crf.abi.EUNSUPPORTED
    ctx.close()
