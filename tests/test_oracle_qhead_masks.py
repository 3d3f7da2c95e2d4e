"""Pins of the oracle's query-head-granular masks (Sec. 3.3: query-head candidates, a KV head
kept whenever one of its query heads is; Table 1: 64 query-head candidates per 70B layer).

The greedy's cost of a query head is its marginal FLOPs with the closure applied first (Eq.
flop-attn: 2 d d_h per Q block and per O block, plus 4 d d_h for the K and V rows when its
group has no kept head yet). Hand-derived cases below follow from that reading; one of them
separates it from ordering by a head's own cost."""
from fractions import Fraction

import numpy as np
import pytest

import synth
from oracle import forward as fw
from oracle import ledger, maskc, pack, weights

SMALL = synth.ModelShape(L=1, d=64, Hq=4, Hkv=2, dh=16, df=4, vocab=0, chan_unit=1)


def _scores(q, ch):
    return np.array([list(q) + list(ch)], dtype=np.uint32)


def test_small_shape_costs():
    # Eq. flop-attn / flop-mlp at d = 64, d_h = 16: Q block + O block = 2*64*16*2
    assert ledger.qhead_cost(SMALL) == 4096
    assert ledger.kv_cost(SMALL) == 4096
    assert ledger.chan_unit_cost(SMALL) == 384
    assert ledger.dense_layer_flops(SMALL) == 4 * 4096 + 2 * 4096 + 4 * 384


def test_closure_cost_decides_the_order():
    # budget 0.75 of 26,112 = 19,584. Forced: head 0 (+ KV 0) = 8,192 and channel 0 = 384.
    # Head 1 shares KV 0 (4,096 for score 60) and beats head 2 (8,192 with KV 1 for 95):
    # 60/4096 > 95/8192. After it 6,912 are left: heads 2 and 3 no longer fit, the three
    # channels do. Ordering by a head's own cost alone would take head 2 instead.
    m = maskc.compile_mask_qheads(SMALL, _scores([100, 60, 95, 0], [1, 0, 0, 0]), [0], 0.75, 0.75, 0.75)
    assert m.keep_qheads == [[0, 1]]
    assert m.keep_groups == [[0]]
    assert m.keep_units == [[0, 1, 2, 3]]
    assert m.info["budget_flops"] == 19584
    assert m.info["total_flops"] == 2 * 4096 + 4096 + 4 * 384 == 13824


def test_second_group_does_not_fit():
    # heads scored far above channels: forced head 3 (+ KV 1), then head 2 at 4,096; head 1
    # would open KV 0 (8,192) and overflow 19,584, so the channels fill the rest.
    m = maskc.compile_mask_qheads(SMALL, _scores([10**9, 10**9 + 1, 10**9 + 2, 10**9 + 3], [3, 2, 1, 0]),
                                  [0], 0.75, 0.75, 0.75)
    assert m.keep_qheads == [[2, 3]]
    assert m.keep_groups == [[1]]
    assert m.keep_units == [[0, 1, 2, 3]]
    assert m.info["total_flops"] == 13824


def test_ratio_tie_goes_to_the_query_head():
    # budget 0.49: b = floor(fixed(0.49) * 26,112 / 2^24) = 12,794; forced head 0 (+ KV 0) and
    # channel 0 leave 4,218. Head 1 (4,096 / 4,096) and channel 1 (384 / 384) tie at ratio 1;
    # the head goes first and then nothing else fits, while channel-first would admit the
    # three channels and no head.
    m = maskc.compile_mask_qheads(SMALL, _scores([10**6, 4096, 0, 0], [10**5, 384, 0, 0]), [0], 0.49, 0.49, 0.49)
    assert m.info["budget_flops"] == 12794
    assert m.keep_qheads == [[0, 1]] and m.keep_units == [[0]]


def _layer1_budget():
    return int(Fraction(57, 100) * ledger.dense_layer_flops(synth.LAYER1))  # floor(0.57 F) = 3,212,574


def test_layer1_heads_first_closed_form():
    # every head scored above every channel: all 8 heads and both KV heads (10 x 131,072),
    # then the highest-scored channels while they fit: k = floor((B - 1,310,720) / 3,072)
    sh = synth.LAYER1
    perm = np.random.default_rng(5).permutation(sh.df)
    sc = _scores([2**31 + h for h in range(sh.Hq)], perm)
    m = maskc.compile_mask_qheads(sh, sc, [123], 0.57, 0.35, 0.85)
    B = _layer1_budget()
    assert B == 3212574 and m.info["budget_flops"] == B
    k = (B - 10 * 131072) // 3072
    assert k == 619
    assert m.keep_qheads == [list(range(8))] and m.keep_groups == [[0, 1]]
    assert m.keep_chans == [sorted(np.argsort(-perm, kind="stable")[:k].tolist())]
    assert m.info["total_flops"] == 10 * 131072 + k * 3072


def test_layer1_channels_first_closed_form():
    # channels scored far above heads: the forced best head with its KV head (262,144), then
    # channels while they fit (960 of them leave 1,310 < one more head's 131,072)
    sh = synth.LAYER1
    perm = np.random.default_rng(6).permutation(sh.df)
    qs = [5, 900, 7, 3, 1000, 2, 8, 1]
    m = maskc.compile_mask_qheads(sh, _scores(qs, 2**31 + perm), [9], 0.57, 0.35, 0.85)
    k = (_layer1_budget() - 262144) // 3072
    assert k == 960
    assert m.keep_qheads == [[4]] and m.keep_groups == [[1]]
    assert m.keep_chans == [sorted(np.argsort(-perm, kind="stable")[:k].tolist())]


@pytest.mark.parametrize("seed", [1, 2, 3, 4])
def test_one_head_per_group_reduces_to_group_masks(seed):
    # g = 1: a head's marginal cost is always a whole group's, so query-head and group
    # candidates coincide and both compilers must agree (the group compiler is pinned on
    # its own by the single-layer closed form and a library sort)
    sh = synth.ModelShape(L=6, d=128, Hq=4, Hkv=4, dh=32, df=256, vocab=0, chan_unit=32)
    sc = synth.mask_scores_u32(seed, sh.L, sh.Hq + sh.n_chan_units)
    tg = synth.layer_target_u24(seed, sh.L)
    for budget, lo, hi in ((0.57, 0.35, 0.85), (0.4, 0.3, 0.6)):
        a = maskc.compile_mask_qheads(sh, sc, tg, budget, lo, hi)
        b = maskc.compile_mask(sh, sc, tg, budget, lo, hi)
        assert a.keep_groups == b.keep_groups and a.keep_units == b.keep_units
        assert a.keep_qheads == b.keep_groups
        assert a.info["layer_flops"] == b.info["layer_flops"]


CASES = [(synth.LLAMA3_8B, 1000), (synth.LLAMA3_8B, 1003), (synth.LLAMA3_70B, 1001), (synth.tiny_shape(L=7), 5)]


def _compile(sh, seed):
    sc = synth.mask_scores_u32(seed, sh.L, sh.Hq + sh.n_chan_units)
    return maskc.compile_mask_qheads(sh, sc, synth.layer_target_u24(seed, sh.L))


@pytest.mark.parametrize("sh,seed", CASES)
def test_closure_budget_and_maximality(sh, seed):
    m = _compile(sh, seed)
    B, cap = m.info["budget_flops"], m.info["layer_cap"]
    # closure: the kept KV heads are exactly the groups of the kept query heads
    for layer in range(sh.L):
        assert m.keep_groups[layer] == sorted({h // sh.g for h in m.keep_qheads[layer]})
        assert len(m.keep_qheads[layer]) >= 1 and len(m.keep_units[layer]) >= 1
    assert maskc.closure_holds(sh, maskc.expand(sh, m))
    # ledger recount and budget
    lf = [ledger.layer_flops(sh, len(q), len(g), len(c))
          for q, g, c in zip(m.keep_qheads, m.keep_groups, m.keep_chans)]
    assert lf == m.info["layer_flops"]
    total = sum(lf)
    assert total == m.info["total_flops"] == ledger.mask_flops(sh, m.keep_groups, m.keep_chans, m.keep_qheads)
    assert total <= B
    # maximal: no further candidate (with its closure) fits the budget and its layer's cap
    for layer in range(sh.L):
        kq, kg = set(m.keep_qheads[layer]), set(m.keep_groups[layer])
        for h in range(sh.Hq):
            if h not in kq:
                c = ledger.qhead_cost(sh) + (0 if h // sh.g in kg else ledger.kv_cost(sh))
                assert total + c > B or lf[layer] + c > cap[layer]
        if len(m.keep_units[layer]) < sh.n_chan_units:
            c = ledger.chan_unit_cost(sh)
            assert total + c > B or lf[layer] + c > cap[layer]


def test_70b_candidate_count_and_ragged_groups():
    sh = synth.LLAMA3_70B
    assert ledger.paper_candidate_count(sh) == sh.L * (sh.Hq + sh.n_chan_units) == 7360
    m = _compile(sh, 1000)
    ragged = sum(1 for layer in range(sh.L) for j in m.keep_groups[layer]
                 if sum(1 for h in m.keep_qheads[layer] if h // sh.g == j) < sh.g)
    assert ragged > 0  # the workload exercises groups with fewer than g kept heads


# --------------------------------------------------------------------------
# Forward with query-head masks
# --------------------------------------------------------------------------

def _steps(sh, n, seed=11):
    return synth.bf16_to_f32(synth.step_inputs_bf16(seed, n, 1, sh.d)[:, 0])


def _ragged_mask(sh):
    # layer 0: one head of group 0 and both of group 1; layer 1: only head 3; layer 2: heads 0, 2
    q = [[1, 2, 3], [3], [0, 2]][:sh.L]
    u = [[0, 3, 5, 11], [2], [1, 4, 6, 7, 8]][:sh.L]
    return maskc.explicit_qheads(sh, q, u)


@pytest.mark.parametrize("dtype,tol", [(np.float64, 1e-12), (np.float32, 2e-5)])
def test_qhead_mask_as_zero_equals_compacted(dtype, tol):
    sh = synth.tiny_shape(L=3)
    m = _ragged_mask(sh)
    assert m.keep_groups == [[0, 1], [1], [0, 1]]
    x = _steps(sh, 5)
    Xz = fw.decode(sh, m, x, 9, 7, dtype=dtype)
    Xc = fw.decode(sh, m, x, 9, 7, compact=True, dtype=dtype)
    assert np.linalg.norm(Xz - Xc) <= tol * np.linalg.norm(Xz)
    # whole-group masks with the same KV heads differ: the dropped heads matter
    Xg = fw.decode(sh, maskc.explicit(sh, m.keep_groups, m.keep_units), x, 9, 7, dtype=dtype)
    assert np.linalg.norm(Xg - Xz) > 1e-3 * np.linalg.norm(Xz)


def test_planted_query_to_kv_map_mistake_is_caught():
    # the compacted step with the group-granular map (kept-head index // g) instead of each
    # head's own group must fail the mask-as-zero equality
    sh = synth.tiny_shape(L=1)
    m = maskc.explicit_qheads(sh, [[1, 2, 3]], [[0, 1]])
    x = _steps(sh, 2).astype(np.float64)
    want = fw.decode(sh, m, x, 6, 7, dtype=np.float64)
    lq = weights.gen_layer(sh, 0)
    P = fw.compact_weights(sh, lq, m.keep_groups[0], m.keep_chans[0], np.float64, m.keep_qheads[0])
    assert P["gmap"] == [0, 1, 1]
    Kc, Vc = fw.prior_cache(sh, 0, 7, 6, m.keep_groups[0], np.float64)
    got, _, _ = fw.layer_step_compact(sh, P, x[0], Kc, Vc, 6)
    assert np.allclose(got, want[0], rtol=1e-12, atol=1e-12)
    P["gmap"] = [i // sh.g for i in range(3)]
    bad, _, _ = fw.layer_step_compact(sh, P, x[0], Kc, Vc, 6)
    assert not np.allclose(bad, want[0], rtol=1e-6, atol=1e-6)


def test_all_heads_of_kept_groups_is_the_group_mask():
    sh = synth.tiny_shape(L=2)
    groups, units = [[1], [0, 1]], [[2, 3], [0, 9]]
    mq = maskc.explicit_qheads(sh, [[2, 3], [0, 1, 2, 3]], units)
    mg = maskc.explicit(sh, groups, units)
    x = _steps(sh, 3).astype(np.float64)
    assert np.array_equal(fw.decode(sh, mq, x, 5, 7, dtype=np.float64), fw.decode(sh, mg, x, 5, 7, dtype=np.float64))


def test_dropped_head_acts_only_through_its_o_columns():
    # with the O columns of dropped heads zero, their Q rows cannot reach the output:
    # restoring those Q rows leaves the step unchanged, restoring the O columns does not
    sh = synth.tiny_shape(L=1)
    lq = weights.gen_layer(sh, 0)
    kq, kg, kc = [1, 2], [0, 1], list(range(0, 192, 3))
    W = weights.dense_zeroed(sh, lq, kg, kc, np.float64, kq)
    full = weights.dense_zeroed(sh, lq, [0, 1], list(range(sh.df)), np.float64)
    x = _steps(sh, 1)[0].astype(np.float64)
    Kc, Vc = fw.prior_cache(sh, 0, 7, 4, None, np.float64)
    base, _, _ = fw.layer_step(sh, W, x, Kc, Vc, 4)
    W2 = dict(W, q=full["q"])
    same, _, _ = fw.layer_step(sh, W2, x, Kc, Vc, 4)
    assert np.array_equal(base, same)
    W3 = dict(W, o=full["o"])
    diff, _, _ = fw.layer_step(sh, W3, x, Kc, Vc, 4)
    assert not np.allclose(base, diff)


def test_qhead_prefill_equals_stepwise_decode():
    sh = synth.tiny_shape(L=2)
    m = _ragged_mask(sh)
    X = _steps(sh, 6).astype(np.float64)
    Xp, _ = fw.prefill(sh, m, X, dtype=np.float64)
    Xd = fw.decode(sh, m, X, 0, 7, dtype=np.float64)
    assert np.allclose(Xp, Xd, rtol=1e-10, atol=1e-10)


def test_ragged_panels_launch_the_ledger_flops():
    sh = synth.tiny_shape(L=3)
    m = _ragged_mask(sh)
    panels = [pack.pack_layer(sh, weights.gen_layer(sh, layer), m.keep_groups[layer], m.keep_chans[layer],
                              m.keep_qheads[layer]) for layer in range(sh.L)]
    assert [p["qkv_w"].shape[0] for p in panels] == [(3 + 4) * sh.dh, (1 + 2) * sh.dh, (2 + 4) * sh.dh]
    assert [p["o_w"].shape[1] for p in panels] == [3 * sh.dh, sh.dh, 2 * sh.dh]
    assert ledger.launched_flops(panels) == ledger.mask_flops(sh, m.keep_groups, m.keep_chans, m.keep_qheads)
