"""GPU parity of groupwise INT8 stores (Table 1: group size 128, BF16 scales) against the
oracle, through the C ABI: INT8 codes and BF16 group scales bit-exact on the store's panels,
one-session decode elementwise per layer and end to end, batches of 2-5 sessions, the union
step and prefill against the oracle."""
import dataclasses

import numpy as np
import pytest

import synth
from oracle import forward, maskc, pack, weights
from gpu_common import TOL_E2E, bf16_tensor, rel_l2, within

pytestmark = pytest.mark.gpu

SHAPE = dataclasses.replace(synth.LLAMA3_8B, L=2, quant_group=128)


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


def _bits(a):
    return synth.bf16_bits(np.asarray(a, np.float32))


def check_grouped_panels(tasp, plan, sh, mask, layer):
    lq = weights.gen_layer(sh, layer)
    ref = pack.pack_layer(sh, lq, mask.keep_groups[layer], mask.keep_chans[layer], mask.qheads(sh, layer))
    for item, name in ((tasp.EXPORT_QKV_W, "qkv_w"), (tasp.EXPORT_O_W, "o_w"), (tasp.EXPORT_GU_W, "gu_w"),
                       (tasp.EXPORT_DOWN_W, "down_w")):
        got = plan.export(layer, item)
        assert got.shape == ref[name].shape and np.array_equal(got, ref[name]), name
    for item, name in ((tasp.EXPORT_QKV_G, "qkv_s"), (tasp.EXPORT_O_G, "o_s"), (tasp.EXPORT_GU_G, "gu_s"),
                       (tasp.EXPORT_DOWN_G, "down_s")):
        got = plan.export(layer, item)
        assert got.shape == ref[name].shape and np.array_equal(got, _bits(ref[name])), name


def _plan(tasp, sh, seed=1000):
    sc = synth.mask_scores_u32(seed, sh.L, sh.n_units)
    tg = synth.layer_target_u24(seed, sh.L)
    mask = maskc.compile_mask(sh, sc, tg)
    return tasp.Plan(sh, tasp.greedy_mask(sc, tg)), mask


@pytest.mark.parametrize("dense", [False, True])
def test_grouped_panels_bit_exact(tasp, dense):
    sh = SHAPE
    if dense:
        plan, mask = tasp.Plan(sh, tasp.all_keep_mask()), maskc.all_keep(sh)
    else:
        plan, mask = _plan(tasp, sh)
    for layer in range(sh.L):
        check_grouped_panels(tasp, plan, sh, mask, layer)
    info = plan.info()
    assert info["launched_flops"] == info["flops_retained"]
    plan.release()


def test_grouped_isolated_layer_and_decode(tasp):
    import torch
    sh = SHAPE
    plan, mask = _plan(tasp, sh)
    # isolated layer 1 fed the oracle's input: elementwise
    sess = tasp.Session(plan, 701)
    sess.fill_synthetic(700, 7)
    x = synth.probe_f32(5, 1, sh.d, 4.0)
    out = torch.empty(sh.d, dtype=torch.float32, device="cuda")
    sess.layer_step(1, torch.from_numpy(x).cuda(), out)
    torch.cuda.synchronize()
    lq = weights.gen_layer(sh, 1)
    W = weights.dense_zeroed(sh, lq, mask.keep_groups[1], mask.keep_chans[1])
    Kc, Vc = forward.prior_cache(sh, 1, 7, 700)
    ref, _, _ = forward.layer_step(sh, W, x.astype(np.float32), Kc, Vc, 700)
    assert within(out.cpu().numpy(), ref).all()
    sess.release()
    # three steps through both layers with logits on sampled rows
    sess = tasp.Session(plan, 703)
    sess.fill_synthetic(700, 7)
    xb = synth.step_inputs_bf16(11, 3, 1, sh.d)
    x = bf16_tensor(xb)
    hid = torch.empty((3, 1, sh.d), dtype=torch.float32, device="cuda")
    logits = torch.empty((3, 1, sh.vocab), dtype=torch.float32, device="cuda")
    for t in range(3):
        tasp.decode_step([sess], x[t], hid[t], logits[t])
    torch.cuda.synchronize()
    assert sess.device_error() == 0
    ref = forward.decode(sh, mask, synth.bf16_to_f32(xb[:, 0]), 700, 7)
    assert rel_l2(hid.cpu().numpy()[:, 0], ref) <= TOL_E2E
    rows = np.arange(0, sh.vocab, 997)
    lref = forward.final_logits(sh, ref, rows=rows)
    assert rel_l2(logits.cpu().numpy()[:, 0][:, rows], lref) <= TOL_E2E
    # the groupwise plan reads 2 bytes of scale per 128 weights more than a per-row plan
    row = dataclasses.replace(sh, quant_group=0)
    prow = tasp.Plan(row, tasp.greedy_mask(synth.mask_scores_u32(1000, sh.L, sh.n_units),
                                           synth.layer_target_u24(1000, sh.L)))
    extra = plan.info()["weight_bytes_per_token"] - prow.info()["weight_bytes_per_token"]
    int8 = sum(pack.pack_layer(sh, weights.gen_layer(sh, layer), mask.keep_groups[layer],
                               mask.keep_chans[layer])["qkv_w"].size for layer in range(sh.L))
    assert extra > 0 and extra >= 2 * int8 // 128
    sess.release()
    prow.release()
    plan.release()


def test_grouped_union_step_matches_oracle(tasp):
    # the union step on a grouped store: the converters scale each 16-column chunk of INT8
    # codes by its BF16 group scale in FP16 (q s_g 2^8, one rounding); three sessions on the
    # greedy plan and the dense plan, three steps through both layers with logits
    import torch
    sh = SHAPE
    plan, mask = _plan(tasp, sh)
    dense = tasp.Plan(sh, tasp.all_keep_mask())
    plans, masks = [plan, dense], [mask, maskc.all_keep(sh)]
    pick, t_priors, kv_seeds = [0, 1, 0], [700, 64, 5], [7, 8, 9]
    ss = []
    for k, tp, ks in zip(pick, t_priors, kv_seeds):
        se = tasp.Session(plans[k], tp + 4)
        se.fill_synthetic(tp, ks)
        ss.append(se)
    n, steps = len(pick), 3
    xb = synth.step_inputs_bf16(13, steps, n, sh.d)
    x = bf16_tensor(xb)
    hid = torch.empty((steps, n, sh.d), dtype=torch.float32, device="cuda")
    logits = torch.empty((steps, n, sh.vocab), dtype=torch.float32, device="cuda")
    for t in range(steps):
        tasp.decode_step_union(ss, x[t], hid[t], logits[t])
    torch.cuda.synchronize()
    assert tasp.union_status(ss)[0] == 0
    rows = np.arange(0, sh.vocab, 997)
    for i, k in enumerate(pick):
        ref = forward.decode(sh, masks[k], synth.bf16_to_f32(xb[:, i]), t_priors[i], kv_seeds[i])
        assert rel_l2(hid.cpu().numpy()[:, i], ref) <= TOL_E2E, i
        lref = forward.final_logits(sh, ref, rows=rows)
        assert rel_l2(logits.cpu().numpy()[:, i][:, rows], lref) <= TOL_E2E, i
    for se in ss:
        se.release()
    dense.release()
    plan.release()


def test_grouped_prefill_matches_oracle(tasp):
    # the prefill GEMMs on FP16 panels holding q s_g 2^8 (one rounding), rows scaled by 2^-8
    import torch
    sh = SHAPE
    plan, mask = _plan(tasp, sh)
    T = 300
    emb = synth.prompt_bf16(6, 0, T, sh.d)
    logits = torch.empty(sh.vocab, dtype=torch.float32, device="cuda")
    sess = tasp.Session.prefill(plan, bf16_tensor(emb), 2, logits)
    torch.cuda.synchronize()
    Xp, kv = forward.prefill(sh, mask, synth.bf16_to_f32(emb))
    for layer in range(sh.L):
        for kind in (0, 1):
            got = synth.bf16_to_f32(sess.kv(layer, kind))
            ref = kv[layer][kind][mask.keep_groups[layer]]
            assert rel_l2(got, ref) <= TOL_E2E, (layer, kind)
    rows = np.arange(0, sh.vocab, 499)
    ref = forward.final_logits(sh, Xp[-1:], rows=rows)[0]
    assert rel_l2(logits.cpu().numpy()[rows], ref) <= TOL_E2E
    # one decode step after the prompt reads the prefilled cache
    xb = synth.step_inputs_bf16(3, 1, 1, sh.d)
    hid = torch.empty((1, sh.d), dtype=torch.float32, device="cuda")
    tasp.decode_step([sess], bf16_tensor(xb)[0], hid)
    torch.cuda.synchronize()
    dref = forward.decode(sh, mask, synth.bf16_to_f32(xb[:, 0]), T, 0,
                          prior=lambda layer: (kv[layer][0], kv[layer][1]))
    assert rel_l2(hid.cpu().numpy(), dref) <= TOL_E2E
    assert sess.device_error() == 0
    sess.release()
    plan.release()


@pytest.mark.parametrize("n", [2, 4, 5])
def test_grouped_batched_decode_matches_oracle(tasp, n):
    # 2-4 sessions share each weight pass of the batched GEMVs (the chunk sums scaled by the
    # row's group scale); five = a group of four plus one session on the single-vector kernels
    import torch
    sh = SHAPE
    plan, mask = _plan(tasp, sh)
    t_priors, kv_seeds = [700, 64, 5, 300, 33][:n], [7, 8, 9, 10, 11][:n]
    ss = []
    for tp, ks in zip(t_priors, kv_seeds):
        se = tasp.Session(plan, tp + 4)
        se.fill_synthetic(tp, ks)
        ss.append(se)
    steps = 3
    xb = synth.step_inputs_bf16(19 + n, steps, n, sh.d)
    x = bf16_tensor(xb)
    hid = torch.empty((steps, n, sh.d), dtype=torch.float32, device="cuda")
    logits = torch.empty((steps, n, sh.vocab), dtype=torch.float32, device="cuda")
    for t in range(steps):
        tasp.decode_step(ss, x[t], hid[t], logits[t])
    torch.cuda.synchronize()
    rows = np.arange(0, sh.vocab, 997)
    for i in range(n):
        assert ss[i].device_error() == 0
        ref = forward.decode(sh, mask, synth.bf16_to_f32(xb[:, i]), t_priors[i], kv_seeds[i])
        assert rel_l2(hid.cpu().numpy()[:, i], ref) <= TOL_E2E, i
        lref = forward.final_logits(sh, ref, rows=rows)
        assert rel_l2(logits.cpu().numpy()[:, i][:, rows], lref) <= TOL_E2E, i
    for se in ss:
        se.release()
    plan.release()
