"""The seeded generator: determinism, distribution, recipes (no method arithmetic involved)."""
import numpy as np
import torch

import synth


def test_deterministic_and_keyed():
    a = synth.normal((1000,), "x", 3)
    assert torch.equal(a, synth.normal((1000,), "x", 3))
    assert not torch.equal(a, synth.normal((1000,), "x", 4))
    assert not torch.equal(a, synth.normal((1000,), "y", 3))
    assert not torch.equal(a, synth.normal((1000,), "x", 3, seed=1))


def test_unit_variance_and_bounds():
    z = synth.normal((400000,), "stats", 0)
    assert abs(z.mean().item()) < 0.01 and abs(z.std().item() - 1) < 0.01
    assert z.abs().max().item() < 3.47


def test_prefix_stability():
    # element i depends only on (key, i): a longer draw extends a shorter one
    assert torch.equal(synth.normal((100,), "p", 0), synth.normal((300,), "p", 0)[:100])


def test_page_permutation_is_permutation():
    p = synth.page_permutation(1000)
    assert sorted(p.tolist()) == list(range(1000))


def test_adapter_versions_perturb_by_layer():
    cfg, lc = synth.TINY, synth.LORA_TINY
    v0 = synth.adapter_version(cfg, lc, 0, 3)
    v1 = synth.adapter_version(cfg, lc, 1, 3)
    dA = (v1["q"][0].float() - v0["q"][0].float()).std().item()
    assert 0.015 < dA < 0.025        # 0.005 * (1 + 3)


def test_batch_plan_ranges():
    ns, wins, gaps = synth.batch_plan(synth.QWEN7B, 8)
    for n, (s, e), g in zip(ns, wins, gaps):
        assert 2048 <= n <= 16384 and 0 <= s < e <= 28 and e - s <= 4 and 1 <= g <= 4
