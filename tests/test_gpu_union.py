"""GPU parity of the union-of-masks decode step: sessions on different plans of one
store in one step, every weight row read once for all of them on the tensor cores.

Each session must match the oracle's decode of that session alone under its own mask
(the mask-as-zero forward of Sec. 3), and agree with the per-plan decode path. Covered:
three kinds of plan (a greedy mask, the dense fallback, an explicit ragged mask), the
largest step (16 sessions), ragged contexts, the 8B widths with all five masks plus the
dense plan, logits, the 70B widths with 16 sessions, bit-identical repeats and panel
layouts, and the argument errors.
"""
import dataclasses

import numpy as np
import pytest

import synth
from oracle import forward, maskc
from gpu_common import TOL_E2E, bf16_tensor, lib_plan, oracle_mask, rel_l2, within

pytestmark = pytest.mark.gpu

# Relative L2 between the union step and the per-plan step of the same session. The union
# step feeds the projections FP16 activations (11 significant bits after a power-of-two
# scale, relative rounding <= 2^-12) where the per-plan GEMVs use 15-bit block-scaled
# digits, and it sums in another order; where a key or value lands next to a BF16 rounding
# boundary of the KV cache the two caches then hold neighbouring BF16 values. A wrong
# session, mask or position differs at O(0.1-1).
TOL_UNION = 5e-3


@pytest.fixture(scope="module")
def tasp():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_29499_gb300 import build
    build.build()
    from paper_2609_29499_gb300 import tasp as t
    t.load()
    torch.cuda.set_device(0)
    return t


def _make(tasp, plans, t_priors, kv_seeds, steps):
    ss = []
    for i, (pl, tp, ks) in enumerate(zip(plans, t_priors, kv_seeds)):
        s = tasp.Session(pl, tp + steps + 3 * i)  # capacities (KV row strides) differ
        s.fill_synthetic(tp, ks)
        ss.append(s)
    return ss


def _run_union(tasp, ss, xb, vocab=0):
    import torch
    S, n, d = xb.shape
    x = bf16_tensor(xb)
    hid = torch.empty((S, n, d), dtype=torch.float32, device="cuda")
    lg = torch.empty((S, n, vocab), dtype=torch.float32, device="cuda") if vocab else None
    for t in range(S):
        tasp.decode_step_union(ss, x[t], hid[t], lg[t] if vocab else None)
    torch.cuda.synchronize()
    return hid.cpu().numpy(), (lg.cpu().numpy() if vocab else None)


def _run_per_plan(tasp, ss, xb, vocab=0):
    import torch
    S, n, d = xb.shape
    x = bf16_tensor(xb)
    hid = torch.empty((S, n, d), dtype=torch.float32, device="cuda")
    lg = torch.empty((S, n, vocab), dtype=torch.float32, device="cuda") if vocab else None
    for t in range(S):
        for i, s in enumerate(ss):
            tasp.decode_step([s], x[t, i:i + 1], hid[t, i:i + 1], lg[t, i:i + 1] if vocab else None)
    torch.cuda.synchronize()
    return hid.cpu().numpy(), (lg.cpu().numpy() if vocab else None)


def _oracle(shape, masks, xb, t_priors, kv_seeds):
    """Oracle decode of every session alone under its own mask: [S, n, d]."""
    X = synth.bf16_to_f32(xb)
    out = np.empty_like(X)
    groups = {}
    for i, m in enumerate(masks):
        groups.setdefault(id(m), (m, []))[1].append(i)
    for m, idx in groups.values():
        out[:, idx] = forward.decode_sessions(shape, m, X[:, idx], [t_priors[i] for i in idx],
                                              [kv_seeds[i] for i in idx])
    return out


@pytest.fixture(scope="module")
def layer1_plans(tasp):
    wl = synth.CFG1
    sh = wl.shape
    groups, units = [[1]], [sorted(set(range(3, 1408, 5)))]
    plans = [lib_plan(tasp, sh, wl.masks[0]), tasp.Plan(sh, tasp.all_keep_mask()),
             tasp.Plan(sh, tasp.explicit_mask(groups, units))]
    masks = [oracle_mask(sh, wl.masks[0]), maskc.all_keep(sh), maskc.explicit(sh, groups, units)]
    yield wl, plans, masks
    for p in plans:
        p.release()


@pytest.mark.parametrize("n", [3, 7, 16])
def test_layer1_union_matches_oracle(tasp, layer1_plans, n):
    wl, plans, masks = layer1_plans
    sh = wl.shape
    steps = 5
    pick = [i % 3 for i in range(n)]
    t_priors = [(128, 40, 1, 77, 100, 9)[i % 6] for i in range(n)]
    kv_seeds = [wl.kv_seed + 11 * i for i in range(n)]
    xb = synth.step_inputs_bf16(wl.x_seed + 31 * n, steps, n, sh.d)
    ss = _make(tasp, [plans[k] for k in pick], t_priors, kv_seeds, steps)
    got, _ = _run_union(tasp, ss, xb)
    err, launches = tasp.union_status(ss)
    assert err == 0 and launches > 0
    for i, s in enumerate(ss):
        assert s.position == t_priors[i] + steps
        assert s.device_error() == 0
    ref = _oracle(sh, [masks[k] for k in pick], xb, t_priors, kv_seeds)
    for i in range(n):
        assert within(got[:, i], ref[:, i]).all(), (i, np.abs(got[:, i] - ref[:, i]).max())
        assert rel_l2(got[:, i], ref[:, i]) <= TOL_E2E
    for s in ss:
        s.release()


def test_layer1_union_agrees_with_per_plan_steps(tasp, layer1_plans):
    wl, plans, _ = layer1_plans
    sh = wl.shape
    steps, n = 4, 6
    pick = [0, 1, 2, 2, 1, 0]
    t_priors, kv_seeds = [128, 3, 64, 90, 17, 128], [5, 6, 7, 8, 9, 10]
    xb = synth.step_inputs_bf16(77, steps, n, sh.d)
    ss = _make(tasp, [plans[k] for k in pick], t_priors, kv_seeds, steps)
    got, _ = _run_union(tasp, ss, xb)
    for s in ss:
        s.release()
    ss = _make(tasp, [plans[k] for k in pick], t_priors, kv_seeds, steps)
    ref, _ = _run_per_plan(tasp, ss, xb)
    for i in range(n):
        assert rel_l2(got[:, i], ref[:, i]) <= TOL_UNION, (i, rel_l2(got[:, i], ref[:, i]))
    for s in ss:
        s.release()


def test_union_errors(tasp, layer1_plans):
    import torch
    wl, plans, _ = layer1_plans
    sh = wl.shape
    ss = _make(tasp, [plans[0]] * 17, [4] * 17, list(range(17)), 2)
    x = torch.zeros((17, sh.d), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(tasp.TaspError):
        tasp.decode_step_union(ss, x)                  # more than 16 sessions
    with pytest.raises(tasp.TaspError):
        tasp.decode_step_union([ss[0], ss[0]], x[:2])  # a session twice
    other = dataclasses.replace(sh, seed=sh.seed + 1)  # another store
    p2 = tasp.Plan(other, tasp.all_keep_mask())
    s2 = tasp.Session(p2, 8)
    with pytest.raises(tasp.TaspError):
        tasp.decode_step_union([ss[0], s2], x[:2])
    s2.release()
    p2.release()
    for s in ss:
        s.release()


def _8b_case(tasp, L):
    sh = dataclasses.replace(synth.LLAMA3_8B, L=L)
    recipes = list(synth.CFG4.masks)
    plans = [lib_plan(tasp, sh, r) for r in recipes] + [tasp.Plan(sh, tasp.all_keep_mask())]
    masks = [oracle_mask(sh, r) for r in recipes] + [maskc.all_keep(sh)]
    pick = [0, 1, 2, 3, 4, 5, 0, 5]
    t_priors = [200, 31, 150, 90, 64, 5, 120, 180]
    kv_seeds = [40 + i for i in range(len(pick))]
    return sh, plans, masks, pick, t_priors, kv_seeds


def test_8b_one_layer_isolated_elementwise(tasp):
    # one layer, first step: both sides start from the same prior cache, so the per-layer
    # elementwise bound applies to every session (five masks and the dense plan)
    sh, plans, masks, pick, t_priors, kv_seeds = _8b_case(tasp, 1)
    xb = synth.step_inputs_bf16(304, 1, len(pick), sh.d)
    ss = _make(tasp, [plans[k] for k in pick], t_priors, kv_seeds, 1)
    got, _ = _run_union(tasp, ss, xb)
    assert tasp.union_status(ss)[0] == 0
    ref = _oracle(sh, [masks[k] for k in pick], xb, t_priors, kv_seeds)
    for i in range(len(pick)):
        assert within(got[0, i], ref[0, i]).all(), (i, np.abs(got[0, i] - ref[0, i]).max())
    for s in ss:
        s.release()
    for p in plans:
        p.release()


def test_8b_two_layers_union_all_masks(tasp):
    # the five masks and the dense plan at the 8B widths (two-layer cut, three steps), with
    # logits: end-to-end bound against the oracle, agreement with the per-plan path
    sh, plans, masks, pick, t_priors, kv_seeds = _8b_case(tasp, 2)
    n, steps = len(pick), 3
    xb = synth.step_inputs_bf16(303, steps, n, sh.d)
    ss = _make(tasp, [plans[k] for k in pick], t_priors, kv_seeds, steps)
    got, lg = _run_union(tasp, ss, xb, sh.vocab)
    assert tasp.union_status(ss)[0] == 0
    for s in ss:
        s.release()
    ref = _oracle(sh, [masks[k] for k in pick], xb, t_priors, kv_seeds)
    for i in range(n):
        assert rel_l2(got[:, i], ref[:, i]) <= TOL_E2E, (i, rel_l2(got[:, i], ref[:, i]))
    ss = _make(tasp, [plans[k] for k in pick], t_priors, kv_seeds, steps)
    ref_pp, lg_pp = _run_per_plan(tasp, ss, xb, sh.vocab)
    for i in range(n):
        assert rel_l2(got[:, i], ref_pp[:, i]) <= TOL_UNION, (i, rel_l2(got[:, i], ref_pp[:, i]))
        assert rel_l2(lg[:, i], lg_pp[:, i]) <= TOL_UNION
    for s in ss:
        s.release()
    for p in plans:
        p.release()


def test_union_is_deterministic_and_ignores_panel_layout(tasp, layer1_plans):
    # the union step sums in a fixed order (no atomics), and it reads the shared store
    # whatever a plan's panel layout: compacted and row-indexed plans give the same bits
    wl, plans, _ = layer1_plans
    sh = wl.shape
    steps, n = 3, 5
    pick = [0, 1, 2, 0, 1]
    t_priors, kv_seeds = [128, 9, 64, 33, 100], [3, 4, 5, 6, 7]
    xb = synth.step_inputs_bf16(91, steps, n, sh.d)
    outs = []
    for _ in range(2):
        ss = _make(tasp, [plans[k] for k in pick], t_priors, kv_seeds, steps)
        outs.append(_run_union(tasp, ss, xb)[0])
        for s in ss:
            s.release()
    assert np.array_equal(outs[0].view(np.uint32), outs[1].view(np.uint32))
    row = lib_plan(tasp, sh, wl.masks[0], panel_mode=tasp.PANELS_ROW_INDEXED)
    ss = _make(tasp, [row if k == 0 else plans[k] for k in pick], t_priors, kv_seeds, steps)
    got = _run_union(tasp, ss, xb)[0]
    for s in ss:
        s.release()
    row.release()
    assert np.array_equal(got.view(np.uint32), outs[0].view(np.uint32))


def test_70b_width_sixteen_sessions_agree_with_per_plan_and_oracle(tasp):
    # the 70B widths (two-layer cut): 16 sessions over the five masks and the dense plan, the
    # down projection's 28,672-long reduction split in K slices; agreement with the per-plan
    # path and with the oracle
    sh = dataclasses.replace(synth.LLAMA3_70B, L=2)
    recipes = list(synth.CFG5.masks)
    plans = [lib_plan(tasp, sh, r) for r in recipes] + [tasp.Plan(sh, tasp.all_keep_mask())]
    n, steps = 16, 2
    pick = [(i * 7) % 6 for i in range(n)]
    t_priors = [64 + 37 * i for i in range(n)]
    kv_seeds = [500 + i for i in range(n)]
    xb = synth.step_inputs_bf16(707, steps, n, sh.d)
    ss = _make(tasp, [plans[k] for k in pick], t_priors, kv_seeds, steps)
    got, _ = _run_union(tasp, ss, xb)
    assert tasp.union_status(ss)[0] == 0
    for s in ss:
        s.release()
    ss = _make(tasp, [plans[k] for k in pick], t_priors, kv_seeds, steps)
    ref, _ = _run_per_plan(tasp, ss, xb)
    for s in ss:
        s.release()
    for i in range(n):
        assert rel_l2(got[:, i], ref[:, i]) <= TOL_UNION, (i, pick[i], rel_l2(got[:, i], ref[:, i]))
    for p in plans:
        p.release()
    # and against the oracle: each plan's sessions decoded under that plan's mask as zeros
    masks = [oracle_mask(sh, r) for r in recipes] + [maskc.all_keep(sh)]
    xf = synth.bf16_to_f32(xb)
    for k, mask in enumerate(masks):
        idx = [i for i in range(n) if pick[i] == k]
        if not idx:
            continue
        want = forward.decode_sessions(sh, mask, xf[:, idx], [t_priors[i] for i in idx], [kv_seeds[i] for i in idx])
        for j, i in enumerate(idx):
            e = rel_l2(got[:, i], want[:, j])
            assert e <= TOL_E2E, (i, k, e)
