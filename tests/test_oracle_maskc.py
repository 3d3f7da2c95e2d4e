"""Pins of the oracle's mask compiler (Sec. 3.3 greedy with dependency closure)."""
import os

import numpy as np
import pytest

import synth
from oracle import ledger, maskc

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _k_layer1():
    with open(os.path.join(GOLD, "flop_ledger_closed_forms.txt")) as f:
        for line in f:
            if line.startswith("layer1_k"):
                return int(line.split()[1])


def _mask(shape, seed, **kw):
    return maskc.compile_mask(shape, synth.mask_scores_u32(seed, shape.L, shape.n_units),
                              synth.layer_target_u24(seed, shape.L), **kw)


def test_layer1_closed_form():
    sh = synth.LAYER1
    sc = synth.mask_scores_u32(1000, 1, sh.n_units)
    m = _mask(sh, 1000)
    assert len(m.keep_groups[0]) == 1
    assert m.keep_groups[0][0] == int(np.argmax(sc[0, :2]))
    assert len(m.keep_chans[0]) == _k_layer1()
    assert m.info["total_flops"] == 655360 + 3072 * 832
    assert m.info["ratio"] == pytest.approx(3211264 / 5636096, abs=0)


def test_layer1_is_top_k_by_score():
    # equal channel costs: score-per-FLOP order is score order (library sort as reference)
    sh = synth.LAYER1
    for seed in (1000, 5, 6):
        sc = synth.mask_scores_u32(seed, 1, sh.n_units)[0, 2:].astype(np.int64)
        m = _mask(sh, seed)
        k = len(m.keep_chans[0])
        top = np.argsort(-sc, kind="stable")[:k]
        assert sorted(top.tolist()) == m.keep_chans[0]


def test_ties_go_to_lower_index():
    sh = synth.tiny_shape(L=1)
    sc = np.full((1, sh.n_units), 1000, dtype=np.uint32)
    m = maskc.compile_mask(sh, sc, np.array([0]), budget=0.3, r_lo=0.1, r_hi=0.9)
    u = m.keep_units[0]
    assert u == list(range(len(u)))  # a prefix of the channel units


@pytest.mark.parametrize("shape,seeds", [(synth.LLAMA3_8B, synth.MASK_SEEDS), (synth.LLAMA3_70B, synth.MASK_SEEDS[:2]),
                                         (synth.tiny_shape(L=6), (1, 2, 3))])
def test_budget_range_maximality_closure(shape, seeds):
    F = ledger.dense_layer_flops(shape)
    costs = ledger.unit_costs(shape)
    umax = max(costs)
    for seed in seeds:
        m = _mask(shape, seed)
        tot = ledger.mask_flops(shape, m.keep_groups, m.keep_chans)
        assert tot == m.info["total_flops"]
        ratio = tot / (shape.L * F)
        assert ratio <= 0.57
        assert ratio >= 0.57 - umax / (shape.L * F)
        for layer in range(shape.L):
            lf = ledger.layer_flops(shape, shape.g * len(m.keep_groups[layer]), len(m.keep_groups[layer]),
                                    len(m.keep_chans[layer]))
            assert lf <= 0.85 * F
            assert lf >= 0.35 * F - umax
            assert len(m.keep_groups[layer]) >= 1 and len(m.keep_units[layer]) >= 1
            # maximal: nothing left out fits under both the global budget and the layer cap
            kept = set(m.keep_groups[layer]) | {shape.Hkv + u for u in m.keep_units[layer]}
            for u in range(shape.n_units):
                if u not in kept:
                    assert (tot + costs[u] > m.info["budget_flops"]) or (lf + costs[u] > m.info["layer_cap"][layer])
        assert maskc.closure_holds(shape, maskc.expand(shape, m))


def test_per_layer_retention_spreads_over_range():
    sh = synth.LLAMA3_70B
    m = _mask(sh, synth.MASK_SEEDS[0])
    F = ledger.dense_layer_flops(sh)
    r = np.array(m.info["layer_flops"]) / F
    assert r.min() < 0.45 and r.max() > 0.75  # targets drawn in [0.35, 0.85], not all at 0.57


def test_closure_predicate_rejects_violations():
    sh = synth.tiny_shape()
    m = _mask(sh, 3)
    sets = maskc.expand(sh, m)
    bad = [dict(s) for s in sets]
    # a query head whose KV head is dropped
    dropped = [j for j in range(sh.Hkv) if j not in sets[0]["kv_heads"]]
    if dropped:
        bad[0] = dict(sets[0], q_heads=sets[0]["q_heads"] | {dropped[0] * sh.g})
        assert not maskc.closure_holds(sh, bad)
    bad = [dict(s) for s in sets]
    bad[0] = dict(sets[0], down=set(list(sets[0]["down"])[1:]))
    assert not maskc.closure_holds(sh, bad)
    bad = [dict(s) for s in sets]
    bad[0] = dict(sets[0], o_heads=set(list(sets[0]["o_heads"])[1:]))
    assert not maskc.closure_holds(sh, bad)


def test_all_keep_is_dense():
    sh = synth.LLAMA3_8B
    m = maskc.all_keep(sh)
    assert ledger.mask_ratio(sh, m.keep_groups, m.keep_chans) == 1.0
    assert all(len(c) == sh.df for c in m.keep_chans)


def test_synthetic_masks_overlap_like_the_papers():
    # the five 70B masks of the mixed-turn workload overlap as the paper's task masks do
    # (pairwise Jaccard of retained units between 0.24 and 0.81: Sec. "Spectral Scoring and Mask
    # Diversity Are Complementary" and the appendix table of task-mask overlaps)
    sh = synth.LLAMA3_70B
    sets = []
    for s in synth.MASK_SEEDS:
        m = maskc.compile_mask(sh, synth.mask_scores_u32(s, sh.L, sh.n_units), synth.layer_target_u24(s, sh.L))
        sets.append({(l, "g", j) for l in range(sh.L) for j in m.keep_groups[l]} |
                    {(l, "c", u) for l in range(sh.L) for u in m.keep_units[l]})
    for i in range(5):
        for j in range(i + 1, 5):
            jac = len(sets[i] & sets[j]) / len(sets[i] | sets[j])
            assert 0.24 <= jac <= 0.81, (i, j, jac)
