"""Host policy of the package against the oracle's restatement of Section 4 (CPU only).

The oracle's policy is pinned to the paper (tests/test_oracle_policy.py); here the package's
independent implementation must take the same decisions, bit for bit, on the same inputs.
"""
import math
import random

import pytest

from oracle import policy as OP
from paper_2609_30884_gb300 import policy as PP

N = 28


def test_first_changed_layer_and_restart_match():
    for m in PP.MODULES:
        for s in range(N):
            assert PP.first_changed_layer(m, s, N) == OP.r_kv(m, s, N)
            assert PP.restart_of([(m, s)], N) == OP.restart_layer(m, s, N)
    # several updates: the shallowest affected one restarts
    assert PP.restart_of([("q", 27), ("v", 20), ("down", 22)], N) == 20
    assert PP.restart_of([("q", 27)], N) is None  # a last-layer query update changes no cache


def test_window_candidates_match():
    for r in range(N):
        assert PP.window_candidates(r, N) == OP.candidate_windows(r, N)


def _conditions(rng, n_cond):
    out = []
    for _ in range(n_cond):
        r = rng.randrange(N)
        h = rng.choice(OP.candidate_windows(r, N))
        d = rng.choice([0.0, 1e-14, rng.uniform(0, 2), rng.uniform(0, 2)])
        out.append((d, r, h))
    return out


@pytest.mark.parametrize("seed", range(6))
def test_sensitivity_matches_eq7(seed):
    rng = random.Random(seed)
    conds = _conditions(rng, rng.choice([1, 5, 20, 80]))
    got = PP.calibrate_sensitivity(conds, N)
    want = OP.sensitivity([d for d, _, _ in conds], [OP.labels(r, h, N) for _, r, h in conds], N)
    assert got == want


@pytest.mark.parametrize("seed", range(8))
def test_risk_window_matches_eq8_eq9(seed):
    rng = random.Random(100 + seed)
    sens = [rng.choice([0.0, rng.uniform(0, 5)]) for _ in range(N)]
    pol = PP.RecoveryPolicy(N, "risk", sensitivity=sens)
    for _ in range(50):
        r = rng.choice([None] + list(range(N)))
        d = [rng.uniform(0, 1) for _ in range(N)]
        if rng.random() < 0.2:  # a risk exactly at the trigger
            l = rng.randrange(N)
            if sens[l] > 0:
                d[l] = 1.0 / sens[l]
        q = OP.risk(sens, d)
        want = OP.plan(r, q)
        got = pol.window(r, d)
        if r is None:
            assert got[0] == got[1]  # reuse, whatever the restart placeholder
            assert want[0] == want[1]
        else:
            assert got == want, (r, got, want)


def test_drift_only_and_fixed_and_baselines():
    pol = PP.RecoveryPolicy(N, "drift_only", threshold=0.5)
    d = [0.0] * N
    d[16] = 0.5
    assert pol.window(14, d) == (14, 17)          # d / threshold = 1 triggers layer 16
    assert pol.window(14, [0.49] * N) == (14, 14)
    assert PP.RecoveryPolicy(N, "fixed", fixed_len=2).window(14) == (14, 16)
    assert PP.RecoveryPolicy(N, "fixed", fixed_len=2).window(27) == (27, 28)
    assert PP.RecoveryPolicy(N, "suffix").window(14) == (14, 28)
    assert PP.RecoveryPolicy(N, "full").window(14) == (0, 28)
    assert PP.RecoveryPolicy(N, "reuse").window(14) == (14, 14)
    with pytest.raises(ValueError):
        PP.RecoveryPolicy(N, "risk", sensitivity=[1.0])
    with pytest.raises(ValueError):
        PP.RecoveryPolicy(N, "drift_only")


def test_trajectory_anchors_match_oracle():
    """32 updates of one middle module: windows and anchors follow the oracle step by step,
    with d_l the whole-state distance between the current version and layer l's anchor."""
    rng = random.Random(7)
    # squared parameter distance between versions a < b: independent increments per version
    inc = [rng.uniform(0.2, 1.0) for _ in range(40)]
    dist2 = lambda a, b: sum(inc[min(a, b):max(a, b)])
    conds = [(math.sqrt(dist2(0, k)), 14, h) for k, h in ((1, 0), (2, 1), (3, 2), (4, 4), (2, 0), (5, 2))]
    sens = PP.calibrate_sensitivity(conds, N)
    pol = PP.RecoveryPolicy(N, "risk", sensitivity=sens)
    anchors = [0] * N
    for t in range(1, 33):
        r = PP.restart_of([("v", 14)], N)
        d = [0.0 if a == t else math.sqrt(dist2(a, t)) for a in pol.anchors]
        table_for = lambda a: [[dist2(a, t)]]  # whole-state squared distance, one cell
        d_or = OP.displacement(anchors, t, table_for)
        assert d == d_or
        w = pol.window(r, d)
        assert w == OP.plan(OP.restart_layer("v", 14, N), OP.risk(sens, d_or))
        pol.commit(w, t)
        anchors = OP.update_anchors(anchors, w, t)
        assert pol.anchors == anchors
        assert pol.fraction(w) == OP.recompute_fraction(w, N)


def test_layer_and_state_displacement_readings_of_eq8():
    """The two readings of d_l (Eq. 8) from a [N][7][2] drift table: per layer, the root of the
    layer's summed weight-space (or parameter-space) squares; over the whole adapter, the root of
    every parameter-space square."""
    import synth
    from oracle import build as obuild, drift as odrift
    HP = PP
    cfg, lc = synth.TINY, synth.LORA_TINY
    a0 = [obuild.layer_adapter(cfg, lc, 0, l).AB for l in range(cfg.n_layers)]
    a2 = [obuild.layer_adapter(cfg, lc, 2, l).AB for l in range(cfg.n_layers)]
    table = odrift.drift_table(a0, a2, synth.MODULES)
    d_w = HP.layer_displacement(table)
    d_p = HP.layer_displacement(table, weight_space=False)
    for l in range(cfg.n_layers):
        want_w = math.sqrt(sum(odrift.dense_sq(*a0[l][m], *a2[l][m]) for m in lc.modules))
        want_p = math.sqrt(sum(odrift.param_sq(*a0[l][m], *a2[l][m]) for m in lc.modules))
        assert d_w[l] == pytest.approx(want_w, rel=1e-10)
        assert d_p[l] == pytest.approx(want_p, rel=1e-12)
    assert HP.state_displacement(table) == pytest.approx(math.sqrt(sum(x * x for x in d_p)), rel=1e-12)
    # identical versions: zero displacement everywhere
    assert HP.layer_displacement(odrift.drift_table(a2, a2, synth.MODULES)) == [0.0] * cfg.n_layers
