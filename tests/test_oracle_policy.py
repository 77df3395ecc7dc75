"""Pins of the host-policy oracle against values the paper prints and worked cases of Eq. 6-9."""
import json
import os

import pytest

from oracle import policy as P

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "policy_paper.json")))
N = GOLD["n_layers"]


def test_onset_eq_s4():
    assert P.r_kv("k", 5, N) == 5 and P.r_kv("v", 5, N) == 5
    for m in ("q", "o", "gate", "up", "down", "mlp"):
        assert P.r_kv(m, 5, N) == 6
        assert P.r_kv(m, N - 1, N) == N          # sentinel: nothing invalidated
    assert P.r_kv("k", N - 1, N) == N - 1
    with pytest.raises(ValueError):
        P.r_kv("embed", 0, N)


@pytest.mark.parametrize("row", GOLD["table_s2"], ids=lambda r: f"{r['module']}-{r['position']}")
def test_table_s2_rows_consistent_with_policy(row):
    s = N - row["suffix_depth"]                  # suffix depth printed in Table S2
    r = P.restart_layer(row["module"], s, N)
    d, b, f = row["dbf"]
    if r is None:
        # nothing invalidated: only direct reuse can be observed, and it always is
        assert row["observed"] == [0] and b == 0 and f == 0
        return
    cands = P.candidate_windows(r, N)
    assert max(cands) == row["suffix_depth"]
    assert set(row["observed"]) <= set(cands)
    if row["module"] in ("q", "mlp"):
        # a one-layer window replaces no affected K/V (Eq. S4): never the first safe window
        assert 1 not in row["observed"]
    assert d + b + f == 9


def test_candidate_windows():
    assert P.candidate_windows(0, N) == [0, 1, 2, 4, 8, 16, 28]
    assert P.candidate_windows(14, N) == [0, 1, 2, 4, 8, 14]
    assert P.candidate_windows(27, N) == [0, 1]


def test_recompute_fractions_printed():
    s = N - 14
    assert 100 * P.recompute_fraction((s, N), N) == pytest.approx(GOLD["exact_suffix_middle_recompute_pct"])
    h = GOLD["fixed_window_layers"]
    assert round(100 * P.recompute_fraction((s, s + h), N), 2) == GOLD["fixed_window_recompute_pct"]


def test_first_safe_is_first_hit_not_monotone():
    cands = [0, 1, 2, 4, 8, 14]
    safe = {0: False, 1: False, 2: True, 4: False, 8: True, 14: True}
    assert P.first_safe(cands, safe.get) == 2
    assert P.first_safe(cands, lambda h: False) is None


def test_labels_eq6():
    assert P.labels(2, 3, 6) == [0, 0, 1, 1, 1, 0]
    assert P.labels(2, 0, 6) == [0] * 6


def test_sensitivity_eq7_order_statistic():
    # layer 0: 20 positive drifts -> floor(0.05*20)+1 = 2nd smallest; layer 1: 19 -> 1st smallest
    d20 = [float(x) for x in range(20, 0, -1)]           # 20..1
    rows = [[1, 1 if i < 19 else 0, 0] for i in range(20)]
    s = P.sensitivity(d20, rows, 3)
    pos1 = sorted(d20[:19])                              # 20..2 -> smallest 2
    assert s[0] == pytest.approx(1 / 2.0)
    assert s[1] == pytest.approx(1 / pos1[0])
    assert s[2] == 0.0                                    # no positives
    # the 1e-12 floor
    assert P.sensitivity([0.0], [[1]], 1) == [1e12]


def test_risk_range_end_plan_eq8_eq9():
    sens = [0.0, 2.0, 0.5, 1.0, 0.0]
    disp = [9.0, 0.6, 1.0, 1.2, 9.0]
    q = P.risk(sens, disp)
    assert q == pytest.approx([0.0, 1.2, 0.5, 1.2, 0.0])
    assert P.range_end(q) == 4
    assert P.plan(1, q) == (1, 4)
    assert P.plan(4, q) == (4, 4)                         # b_t <= r: reuse
    assert P.plan(None, q) == (0, 0)
    assert P.range_end([0.99, 0.5]) is None
    assert P.range_end([1.0]) == 1                        # q >= 1 triggers


def test_anchor_update_only_in_window():
    assert P.update_anchors([0, 0, 1, 1, 2], (1, 3), 5) == [0, 5, 5, 1, 2]
    assert P.update_anchors([3, 3], (1, 1), 5) == [3, 3]


def test_displacement_whole_adapter():
    tables = {0: [[1.0, 3.0], [0.0, 5.0]], 1: [[0.25, 0.0], [0.0, 0.0]]}
    assert P.displacement([0, 1, 2], 2, tables.get) == pytest.approx([3.0, 0.5, 0.0])
