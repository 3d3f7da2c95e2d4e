"""GPU parity of query-head-granular masks (Sec. 3.3: query-head candidates, a KV head kept
whenever one of its heads is) against the oracle, through the C ABI: panels and kept lists
bit-exact, decode and prefill elementwise, compact = row-indexed panels bit for bit, and
union steps that mix query-head plans with whole-group and dense plans."""
import dataclasses

import numpy as np
import pytest

import synth
from oracle import forward, maskc, pack, weights
from gpu_common import TOL_E2E, bf16_tensor, rel_l2, within

pytestmark = pytest.mark.gpu


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


def check_qhead_panels(tasp, plan, shape, mask, layer):
    lq = weights.gen_layer(shape, layer)
    qh = mask.keep_qheads[layer]
    ref = pack.pack_layer(shape, lq, mask.keep_groups[layer], mask.keep_chans[layer], qh)
    assert plan.layer_qheads(layer) == len(qh)
    assert plan.export(layer, tasp.EXPORT_KEEP_QHEADS).tolist() == qh
    assert plan.export(layer, tasp.EXPORT_KEEP_GROUPS).tolist() == mask.keep_groups[layer]
    items = {tasp.EXPORT_QKV_W: "qkv_w", tasp.EXPORT_QKV_S: "qkv_s", tasp.EXPORT_O_W: "o_w",
             tasp.EXPORT_GU_W: "gu_w", tasp.EXPORT_DOWN_W: "down_w"}
    for item, name in items.items():
        got, want = plan.export(layer, item), ref[name]
        assert got.shape == want.shape, name
        assert np.array_equal(got.view(np.uint8) if got.dtype == np.int8 else got.view(np.uint32),
                              want.view(np.uint8) if want.dtype == np.int8 else want.view(np.uint32)), name


def _decode(tasp, plan, sh, t_prior, kv_seed, xb):
    import torch
    S = xb.shape[0]
    sess = tasp.Session(plan, t_prior + S)
    sess.fill_synthetic(t_prior, kv_seed)
    x = bf16_tensor(xb)
    hid = torch.empty((S, 1, sh.d), dtype=torch.float32, device="cuda")
    for t in range(S):
        tasp.decode_step([sess], x[t], hid[t])
    torch.cuda.synchronize()
    assert sess.device_error() == 0
    sess.release()
    return hid.cpu().numpy()[:, 0]


# layer 0 of the single-layer shape (g = 4): group 0 keeps heads 1-3, group 1 keeps 4 and 6
LAYER1_HEADS = [[1, 2, 3, 4, 6]]


@pytest.mark.parametrize("panel_mode", [0, 1])
def test_layer1_partial_groups_decode(tasp, panel_mode):
    wl = synth.CFG1
    sh = wl.shape
    units = [list(range(0, sh.df, 2))]
    mask = maskc.explicit_qheads(sh, LAYER1_HEADS, units)
    plan = tasp.Plan(sh, tasp.explicit_qhead_mask(LAYER1_HEADS, units, panel_mode))
    check_qhead_panels(tasp, plan, sh, mask, 0)
    info = plan.info()
    assert info["launched_flops"] == info["flops_retained"]
    xb = synth.step_inputs_bf16(wl.x_seed, 6, 1, sh.d)
    got = _decode(tasp, plan, sh, wl.t_prior, wl.kv_seed, xb)
    ref = forward.decode(sh, mask, synth.bf16_to_f32(xb[:, 0]), wl.t_prior, wl.kv_seed)
    assert within(got, ref).all(), np.abs(got - ref).max()
    plan.release()


def test_compact_and_row_indexed_partial_groups_agree(tasp):
    wl = synth.CFG1
    sh = wl.shape
    units = [list(range(5, sh.df, 3))]
    xb = synth.step_inputs_bf16(wl.x_seed + 1, 3, 1, sh.d)
    outs = []
    for mode in (0, 1):
        plan = tasp.Plan(sh, tasp.explicit_qhead_mask(LAYER1_HEADS, units, mode))
        outs.append(_decode(tasp, plan, sh, wl.t_prior, wl.kv_seed, xb))
        plan.release()
    assert np.array_equal(outs[0], outs[1])


def test_8b_two_layer_greedy_qhead_mask(tasp):
    # budget 0.3: both layers keep 30 of 32 query heads over all 8 KV groups (partial groups)
    sh = dataclasses.replace(synth.LLAMA3_8B, L=2)
    seed = 1002
    sc = synth.mask_scores_u32(seed, sh.L, sh.Hq + sh.n_chan_units)
    tg = synth.layer_target_u24(seed, sh.L)
    mask = maskc.compile_mask_qheads(sh, sc, tg, 0.3, 0.1, 0.5)
    assert all(len(mask.keep_qheads[l]) < len(mask.keep_groups[l]) * sh.g for l in range(sh.L))
    plan = tasp.Plan(sh, tasp.greedy_qhead_mask(sc, tg, 0.3, 0.1, 0.5))
    for layer in range(sh.L):
        check_qhead_panels(tasp, plan, sh, mask, layer)
    xb = synth.step_inputs_bf16(11, 3, 1, sh.d)
    got = _decode(tasp, plan, sh, 700, 7, xb)
    ref = forward.decode(sh, mask, synth.bf16_to_f32(xb[:, 0]), 700, 7)
    assert rel_l2(got, ref) <= TOL_E2E
    plan.release()


@pytest.mark.parametrize("T", [100, 300])
def test_layer1_partial_groups_prefill(tasp, T):
    import torch
    sh = synth.LAYER1
    units = [list(range(0, sh.df, 2))]
    mask = maskc.explicit_qheads(sh, LAYER1_HEADS, units)
    plan = tasp.Plan(sh, tasp.explicit_qhead_mask(LAYER1_HEADS, units))
    emb = synth.prompt_bf16(5, 0, T, sh.d)
    sess = tasp.Session.prefill(plan, bf16_tensor(emb), 2)
    torch.cuda.synchronize()
    Xp, kv = forward.prefill(sh, mask, synth.bf16_to_f32(emb))
    K = synth.bf16_to_f32(sess.kv(0, 0))
    V = synth.bf16_to_f32(sess.kv(0, 1))
    Kref, Vref = kv[0][0][mask.keep_groups[0]], kv[0][1][mask.keep_groups[0]]
    assert within(K, Kref).all() and within(V, Vref).all()
    # one decode step after the prompt reads the prefilled cache
    xb = synth.step_inputs_bf16(3, 1, 1, sh.d)
    hid = torch.empty((1, sh.d), dtype=torch.float32, device="cuda")
    tasp.decode_step([sess], bf16_tensor(xb)[0], hid)
    torch.cuda.synchronize()
    ref = forward.decode(sh, mask, synth.bf16_to_f32(xb[:, 0]), T, 0,
                         prior=lambda layer: (kv[layer][0], kv[layer][1]))
    assert within(hid.cpu().numpy(), ref).all()
    assert sess.device_error() == 0
    sess.release()
    plan.release()


def _union(tasp, plans, t_priors, kv_seeds, xb):
    import torch
    S, n, d = xb.shape
    ss = []
    for pl, tp, ks in zip(plans, t_priors, kv_seeds):
        s = tasp.Session(pl, tp + S + 1)
        s.fill_synthetic(tp, ks)
        ss.append(s)
    x = bf16_tensor(xb)
    hid = torch.empty((S, n, d), dtype=torch.float32, device="cuda")
    for t in range(S):
        tasp.decode_step_union(ss, x[t], hid[t])
    torch.cuda.synchronize()
    assert tasp.union_status(ss)[0] == 0
    for i, s in enumerate(ss):
        assert s.position == t_priors[i] + S and s.device_error() == 0
        s.release()
    return hid.cpu().numpy()


def test_layer1_union_with_partial_groups_matches_oracle(tasp):
    # one union step over a query-head plan (partial groups), a whole-group plan and the
    # dense plan: each session against the oracle's decode under its own mask
    wl = synth.CFG1
    sh = wl.shape
    units = [list(range(0, sh.df, 2))]
    plans = [tasp.Plan(sh, tasp.explicit_qhead_mask(LAYER1_HEADS, units)),
             tasp.Plan(sh, tasp.explicit_mask([[1]], units)), tasp.Plan(sh, tasp.all_keep_mask())]
    masks = [maskc.explicit_qheads(sh, LAYER1_HEADS, units), maskc.explicit(sh, [[1]], units), maskc.all_keep(sh)]
    pick = [0, 1, 2, 0, 0]
    t_priors, kv_seeds = [128, 40, 77, 9, 300], [5, 6, 7, 8, 9]
    xb = synth.step_inputs_bf16(21, 4, len(pick), sh.d)
    got = _union(tasp, [plans[k] for k in pick], t_priors, kv_seeds, xb)
    for i, k in enumerate(pick):
        ref = forward.decode(sh, masks[k], synth.bf16_to_f32(xb[:, i]), t_priors[i], kv_seeds[i])
        assert within(got[:, i], ref).all(), (i, np.abs(got[:, i] - ref).max())
        assert rel_l2(got[:, i], ref) <= TOL_E2E
    for p in plans:
        p.release()


def test_8b_two_layer_union_of_query_head_plans(tasp):
    # head dim 128: two greedy query-head masks in one union step, against the oracle
    sh = dataclasses.replace(synth.LLAMA3_8B, L=2)
    plans, masks = [], []
    for seed, (budget, lo, hi) in ((1002, (0.3, 0.1, 0.5)), (7, (0.2, 0.05, 0.4))):
        sc = synth.mask_scores_u32(seed, sh.L, sh.Hq + sh.n_chan_units)
        tg = synth.layer_target_u24(seed, sh.L)
        masks.append(maskc.compile_mask_qheads(sh, sc, tg, budget, lo, hi))
        plans.append(tasp.Plan(sh, tasp.greedy_qhead_mask(sc, tg, budget, lo, hi)))
    for m in masks:  # partial groups in every layer: 30/32 heads over 8 groups; 20/6 and 25/8
        assert all(len(m.keep_qheads[l]) < len(m.keep_groups[l]) * sh.g for l in range(sh.L))
    pick, t_priors, kv_seeds = [0, 1, 1, 0], [300, 64, 5, 150], [41, 42, 43, 44]
    xb = synth.step_inputs_bf16(17, 3, len(pick), sh.d)
    got = _union(tasp, [plans[k] for k in pick], t_priors, kv_seeds, xb)
    for i, k in enumerate(pick):
        ref = forward.decode(sh, masks[k], synth.bf16_to_f32(xb[:, i]), t_priors[i], kv_seeds[i])
        assert rel_l2(got[:, i], ref) <= TOL_E2E, (i, rel_l2(got[:, i], ref))
    for p in plans:
        p.release()


def test_8b_two_layer_partial_groups_prefill(tasp):
    # head dim 128: the tcgen05 prefill attention, with dropped heads' outputs skipped
    import torch
    sh = dataclasses.replace(synth.LLAMA3_8B, L=2)
    heads = [[0, 1, 2, 5, 9, 10, 11, 31], [3, 4, 7, 30]]
    units = [[0, 5, 13], [2, 3]]
    mask = maskc.explicit_qheads(sh, heads, units)
    plan = tasp.Plan(sh, tasp.explicit_qhead_mask(heads, units))
    T = 200
    emb = synth.prompt_bf16(6, 0, T, sh.d)
    logits = torch.empty(sh.vocab, dtype=torch.float32, device="cuda")
    sess = tasp.Session.prefill(plan, bf16_tensor(emb), 2, logits)
    torch.cuda.synchronize()
    Xp, kv = forward.prefill(sh, mask, synth.bf16_to_f32(emb))
    for layer in range(sh.L):
        K = synth.bf16_to_f32(sess.kv(layer, 0))
        Kref = kv[layer][0][mask.keep_groups[layer]]
        assert rel_l2(K, Kref) <= TOL_E2E
    rows = np.arange(0, sh.vocab, 499)
    ref = forward.final_logits(sh, Xp[-1:], rows=rows)[0]
    assert rel_l2(logits.cpu().numpy()[rows], ref) <= TOL_E2E
    assert sess.device_error() == 0
    sess.release()
    plan.release()
