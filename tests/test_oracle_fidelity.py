"""Pins of the KL / top-1 / tail-influence oracle against closed forms, libraries and Eq. 4-5."""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F
from scipy.special import rel_entr, softmax

from oracle import fidelity as Fi

RNG = np.random.default_rng(7)


def test_kl_closed_form_two_symbols():
    # p* = (1/2, 1/2), p = (3/4, 1/4): KL = 1/2 log(4/3)
    assert Fi.kl(np.array([0.0, 0.0]), np.array([math.log(3.0), 0.0])) == pytest.approx(
        0.5 * math.log(4.0 / 3.0), rel=1e-14)


def test_kl_self_zero_nonneg_shift_invariant():
    z = RNG.standard_normal((5, 1000)) * 3
    w = z + RNG.standard_normal((5, 1000)) * 0.3
    assert np.all(np.abs(Fi.kl(z, z)) < 1e-13)
    k = Fi.kl(z, w)
    assert np.all(k > 0)
    np.testing.assert_allclose(Fi.kl(z + 17.0, w - 4.0), k, rtol=1e-10)


def test_kl_matches_torch_and_scipy():
    z = RNG.standard_normal((3, 257)) * 2
    w = RNG.standard_normal((3, 257)) * 2
    ref = F.kl_div(torch.log_softmax(torch.tensor(w), -1), torch.log_softmax(torch.tensor(z), -1),
                   reduction="none", log_target=True).sum(-1).numpy()
    np.testing.assert_allclose(Fi.kl(z, w), ref, rtol=1e-12)
    np.testing.assert_allclose(Fi.kl(z, w), rel_entr(softmax(z, -1), softmax(w, -1)).sum(-1),
                               rtol=1e-10)


def test_kl_is_bregman_of_logsumexp():
    """KL(p*||p) = A(z) - A(z*) - <softmax(z*), z - z*> (Section S1.2)."""
    z = RNG.standard_normal(300)
    w = RNG.standard_normal(300)
    A = lambda a: np.log(np.exp(a - a.max()).sum()) + a.max()
    breg = A(w) - A(z) - softmax(z) @ (w - z)
    assert Fi.kl(z, w) == pytest.approx(breg, rel=1e-10)


def test_kl_certificate_holds_and_is_quarter_smooth():
    """KL(p*||p) <= ||z - z*||^2 / 4 for any pair (Eq. 4 via 1/2-smoothness)."""
    for scale in (0.01, 0.3, 3.0):
        z = RNG.standard_normal((200, 64)) * 2
        w = z + RNG.standard_normal((200, 64)) * scale
        bound = 0.25 * np.sum((w - z) ** 2, axis=1)
        assert np.all(Fi.kl(z, w) <= bound + 1e-15)
    # the constant 1/4 is attained in the limit: two equiprobable symbols, opposite shift
    # (KL ~ Var_p(dz) / 2 = eps^2 / 2 = ||dz||^2 / 4)
    eps = 1e-3
    z = np.array([0.0, 0.0])
    w = np.array([eps, -eps])
    assert Fi.kl(z, w) / (0.25 * np.sum((w - z) ** 2)) == pytest.approx(1.0, rel=1e-5)


def test_tail_influence_telescoping_and_certificates():
    n_layers, V = 6, 50
    z = [RNG.standard_normal(V) for _ in range(n_layers + 1)]
    z[-1] = z[-1] * 4            # fresh logits with a clear margin
    T = Fi.tail_influence(z)
    assert T[-1] == 0.0 and np.all(np.diff(T) <= 0)
    for b in range(n_layers + 1):
        # ||z^(b) - z*|| <= T_b (triangle inequality on the telescoped sum)
        assert np.linalg.norm(z[b] - z[-1]) <= T[b] + 1e-12
        assert Fi.kl(z[-1], z[b]) <= Fi.kl_certificate(T[b]) + 1e-12


def test_top1_certificate():
    """T_b < gamma*/2 implies argmax preserved (Eq. 5)."""
    for _ in range(200):
        zs = RNG.standard_normal(30)
        gamma = Fi.margin(zs)
        d = RNG.standard_normal(30)
        d *= 0.999 * (gamma / 2) / np.linalg.norm(d)
        assert Fi.top1_agree(zs, zs + d)


def test_margin_and_top1_ties():
    assert Fi.margin(np.array([1.0, 3.0, 2.5])) == pytest.approx(0.5)
    assert Fi.top1_agree(np.array([1.0, 1.0]), np.array([2.0, 2.0]))
