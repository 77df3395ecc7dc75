"""Failure detection on the GPU without a fault: a bounded wait that nothing completes runs out,
the host reads CRF_ETIMEOUT from crf_check, the report is cleared and the same context keeps
working (a KL from logits against the oracle after the timeout)."""
import time

import numpy as np
import pytest
import torch

import synth
from oracle import fidelity
from tests.gpu_util import KL_ABS

pytestmark = pytest.mark.gpu


def test_bounded_wait_times_out_and_context_stays_usable():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_30884_gb300 as crf
    ctx = crf.Context(0)
    ctx.check()
    t0 = time.time()
    ctx.selftest_timeout()
    with pytest.raises(crf.CrfError) as ei:
        ctx.check()
    assert ei.value.status == crf.abi.ETIMEOUT
    assert time.time() - t0 >= 1.5          # the wait ran to its limit
    ctx.check()                             # the report was cleared
    rows, vocab = 2, 4096
    z_ref = synth.normal((rows, vocab), "zref_fail", 0, 1.0, device="cuda")
    z_cur = z_ref + synth.normal((rows, vocab), "dz_fail", 0, 0.3, device="cuda")
    out = torch.empty(rows, dtype=torch.float32, device="cuda")
    ctx.kl(None, z_ref, z_cur, out, vocab, ctx.kl_workspace(rows, vocab))
    ctx.check()
    want = fidelity.kl(z_ref.double().cpu().numpy(), z_cur.double().cpu().numpy())
    np.testing.assert_allclose(out.double().cpu().numpy(), want, atol=KL_ABS, rtol=0)
