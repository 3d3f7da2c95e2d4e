"""Pins of the per-turn plan choice with the dense fallback (Sec. 3.3, Table 1)."""
import numpy as np
import pytest

from oracle import dispatch


def test_rule_at_the_papers_threshold():
    assert dispatch.choose_plan([0.9, 0.05, 0.05, 0.0, 0.0]) == 0
    assert dispatch.choose_plan([0.05, 0.05, 0.0, 0.0, 0.9]) == 4
    assert dispatch.choose_plan([0.5, 0.3, 0.1, 0.05, 0.05]) == 5   # below tau: dense plan
    assert dispatch.choose_plan([0.85, 0.15, 0, 0, 0]) == 0            # at tau: sparse
    assert dispatch.choose_plan([0.2] * 5) == 5


def test_ties_and_other_thresholds():
    assert dispatch.choose_plan([0.5, 0.5], tau=0.5) == 0
    assert dispatch.choose_plan([0.1, 0.45, 0.45], tau=0.4) == 1
    assert dispatch.choose_plan([0.3, 0.7], tau=0.0) == 1
    assert dispatch.choose_plan([0.3, 0.7], tau=1.0) == 2
    with pytest.raises(ValueError):
        dispatch.choose_plan([0.5, float("nan")])
    with pytest.raises(ValueError):
        dispatch.choose_plan([0.5, 0.5], tau=1.5)


def test_matches_argmax_on_random_distributions():
    rng = np.random.default_rng(3)
    for _ in range(500):
        p = rng.dirichlet(np.full(5, 0.3))
        want = int(np.argmax(p)) if p.max() >= 0.85 else 5
        assert dispatch.choose_plan(p) == want
