"""Host side of the tail-influence sweep (paper_2609_30884_gb300.tail.certificates) against the
oracle's restatement of Eq. 2-5, on synthetic hybrid logits (CPU)."""
import numpy as np

from oracle import fidelity as Fi
from paper_2609_30884_gb300 import tail

RNG = np.random.default_rng(7)


def _hybrid(n_layers=8, V=64, scale=0.3):
    z_star = RNG.standard_normal(V) * 3.0
    # z^(b) drifts away from z* as b falls (more of the cache historical)
    z = [z_star + scale * (n_layers - b) * RNG.standard_normal(V) for b in range(n_layers)] + [z_star]
    return np.stack(z)


def test_certificates_match_oracle_restatement():
    z = _hybrid()
    kl = np.array([Fi.kl(z[-1], z[b]) for b in range(len(z))])
    ts = tail.certificates(z, kl)
    np.testing.assert_allclose(ts.tail, Fi.tail_influence(list(z)), rtol=1e-13, atol=1e-13)
    assert ts.margin == Fi.margin(z[-1])
    assert ts.tail[-1] == 0.0 and ts.kl[-1] == 0.0
    np.testing.assert_array_equal(ts.top1, [Fi.top1_agree(z[-1], z[b]) for b in range(len(z))])
    # with exact KLs both certificates hold at every boundary (Eq. 4, Eq. 5)
    assert ts.kl_certificate_holds.all() and ts.top1_certificate_holds.all()


def test_certificate_flags_detect_a_violation():
    z = _hybrid()
    kl = np.array([Fi.kl(z[-1], z[b]) for b in range(len(z))])
    bad = kl.copy()
    bad[2] = 0.25 * tail.certificates(z, kl).tail[2] ** 2 + 1.0   # above T_b^2 / 4 + slack
    assert not tail.certificates(z, bad).kl_certificate_holds[2]
    # Eq. 5 by contraposition: where the argmax flips, T_b >= gamma*/2. Swap the top two fresh
    # logits at boundary 3 of an otherwise fresh sweep.
    z2 = np.repeat(z[-1:], len(z), axis=0)
    i, j = np.argsort(z2[-1])[-2:]
    z2[3, i], z2[3, j] = z2[-1, j], z2[-1, i]
    ts = tail.certificates(z2, np.zeros(len(z2)))
    assert not ts.top1[3] and ts.top1[[0, 1, 2, 4, 5, 6, 7, 8]].all()
    assert ts.tail[3] >= ts.margin / 2 and ts.top1_certificate_holds.all()
    # the swapped row enters v_2 and v_3: T_0 = T_2 = 2 T_3, and nothing after it
    assert ts.tail[4] == 0.0 and np.isclose(ts.tail[0], 2 * ts.tail[3]) and ts.tail[2] == ts.tail[0]


def test_horizon_counts_from_the_restart():
    z = _hybrid()
    kl = np.array([0.5, 0.4, 0.3, 0.02, 0.05, 0.001, 0.0, 0.0, 0.0])
    ts = tail.certificates(z, kl)
    assert ts.horizon(0, 0.03) == 3
    assert ts.horizon(4, 0.03) == 1
    assert ts.horizon(0, 1e-9) == 6
    assert ts.horizon(8, 0.0) == 0
