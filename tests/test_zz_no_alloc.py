"""The allocation-free KL entry point against the oracle and against the workspace entry point.

Some callers of this library cannot allocate device memory at the moment they need the
first-step fidelity number: a serving loop whose device memory is partitioned once at start-up,
or a C host that has no device allocator of its own. crf_kl_logits_noalloc serves them: its
scratch is a fixed device array inside the library, so the caller passes only the logits and the
output. Every call reuses that array, so two calls in a row must both be right. The cases cover
both edges of the array: all 32 rows, and one row over a vocabulary large enough to need the
largest split count (256). This file is collected last so that a run stopping at the first
failure has already run every other test.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import fidelity
from tests.gpu_util import KL_ABS

pytestmark = pytest.mark.gpu


def _workspace_kl(ctx, z_ref, z_cur):
    out = torch.empty(z_ref.shape[0], dtype=torch.float32, device="cuda:0")
    ws = ctx.kl_workspace(z_ref.shape[0], z_ref.shape[1])
    ctx.kl(None, z_ref, z_cur, out, z_ref.shape[1], ws)
    torch.cuda.synchronize()
    return out.cpu().numpy()


@pytest.mark.parametrize("rows,vocab", [(3, 152064), (32, 151936), (1, 300000)])
def test_noalloc_kl_matches_oracle_twice(rows, vocab):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30884_gb300 as crf
    ctx = crf.Context(0)
    # logits drawn on the host (the generator is device-agnostic) and moved to the device
    z_ref_h = synth.normal((rows, vocab), "noalloc_ref", rows, 2.0)
    z_ref = z_ref_h.to("cuda:0")
    for call in range(2):       # two calls in a row share the fixed scratch
        z_cur_h = z_ref_h + synth.normal((rows, vocab), "noalloc_cur", 10 * rows + call, 0.3 + call)
        z_cur = z_cur_h.to("cuda:0")
        out = torch.full((rows,), float("nan"), dtype=torch.float32, device="cuda:0")
        crf.kl_logits_noalloc(0, z_ref, z_cur, out)
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        want = fidelity.kl(z_ref_h.numpy().astype(np.float64), z_cur_h.numpy().astype(np.float64))
        np.testing.assert_allclose(got, want, atol=KL_ABS, rtol=0)
        # same splits and order as the workspace entry point: the same bits
        np.testing.assert_array_equal(got, _workspace_kl(ctx, z_ref, z_cur))
    ctx.close()


def test_noalloc_kl_rejects_rows_beyond_its_scratch():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30884_gb300 as crf
    too_many = torch.zeros(33, 8, dtype=torch.float32, device="cuda:0")
    out = torch.full((33,), 7.0, dtype=torch.float32, device="cuda:0")
    with pytest.raises(crf.CrfError) as ei:
        crf.kl_logits_noalloc(0, too_many, too_many, out)
    assert ei.value.status == crf.abi.EUNSUPPORTED
    torch.cuda.synchronize()
    assert torch.all(out == 7.0)        # nothing was written
