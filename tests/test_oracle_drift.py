"""Pins of the drift oracle: factored == dense, closed forms, symmetry."""
import numpy as np
import pytest

import synth
from oracle import build, drift

RNG = np.random.default_rng(11)


def _ab(r, i, o, s=1.0):
    return RNG.standard_normal((r, i)) * s, RNG.standard_normal((o, r)) * s


@pytest.mark.parametrize("r,i,o", [(1, 5, 7), (4, 16, 9), (8, 33, 20)])
def test_factored_equals_dense(r, i, o):
    A0, B0 = _ab(r, i, o)
    A1, B1 = A0 + 0.1 * RNG.standard_normal(A0.shape), B0 + 0.1 * RNG.standard_normal(B0.shape)
    assert drift.factored_sq(A0, B0, A1, B1) == pytest.approx(drift.dense_sq(A0, B0, A1, B1), rel=1e-11)


def test_zero_and_symmetry():
    A0, B0 = _ab(4, 10, 12)
    A1, B1 = _ab(4, 10, 12)
    assert drift.factored_sq(A0, B0, A0, B0) == 0.0
    assert drift.param_sq(A0, B0, A0, B0) == 0.0
    assert drift.factored_sq(A0, B0, A1, B1) == pytest.approx(drift.factored_sq(A1, B1, A0, B0), rel=1e-11)
    assert drift.param_sq(A0, B0, A1, B1) == pytest.approx(drift.param_sq(A1, B1, A0, B0))


def test_rank_one_closed_form():
    # B unchanged: ||b a1^T - b a0^T||^2 = ||b||^2 ||a1 - a0||^2
    a0, a1 = RNG.standard_normal((1, 9)), RNG.standard_normal((1, 9))
    b = RNG.standard_normal((6, 1))
    want = float(np.sum(b * b) * np.sum((a1 - a0) ** 2))
    assert drift.factored_sq(a0, b, a1, b) == pytest.approx(want, rel=1e-12)
    assert drift.param_sq(a0, b, a1, b) == pytest.approx(float(np.sum((a1 - a0) ** 2)))


def test_small_drift_no_cancellation():
    """Factored form keeps relative accuracy when the two versions are nearly equal."""
    A0, B0 = _ab(8, 64, 64)
    eps = 1e-7
    dA, dB = eps * RNG.standard_normal(A0.shape), eps * RNG.standard_normal(B0.shape)
    got = drift.factored_sq(A0, B0, A0 + dA, B0 + dB)
    # first-order expansion (exact up to eps^4 terms): ||dB A0 + B0 dA + dB dA||^2
    exact = float(np.sum((dB @ A0 + B0 @ dA + dB @ dA) ** 2))
    assert got == pytest.approx(exact, rel=1e-6)


def test_table_on_synthetic_versions():
    cfg, lc = synth.TINY, synth.LORA_TINY
    a0 = build.adapter(cfg, lc, 0).layers
    a1 = build.adapter(cfg, lc, 1).layers
    to_dict = lambda ls: [l.AB for l in ls]
    t = drift.drift_table(to_dict(a0), to_dict(a1), synth.MODULES)
    td = drift.drift_table(to_dict(a0), to_dict(a1), synth.MODULES, dense=True)
    np.testing.assert_allclose(t, td, rtol=1e-10)
    assert t.shape == (4, 7, 2)
    assert np.all(t[:, 4:] == 0)                       # MLP modules not adapted in this config
    assert np.all(t[:, :4, 1] > 0)
    # perturbation std grows with the layer index (0.005 (1 + l))
    assert t[3, 0, 1] > t[0, 0, 1]
