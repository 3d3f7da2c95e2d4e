"""GPU parity of the decode path against the CPU oracle, through the C ABI.

Single-layer workload: whole-run parity (16 steps). Llama-3-8B / 70B shapes: index
lists and panels bit-exact on sampled layers, isolated layers (fed the oracle's
input) elementwise, and an 8B end-to-end run on final hidden states and sampled
logits. Everything uses the launch configuration of the benchmark.
"""
import numpy as np
import pytest

import synth
from oracle import forward, maskc
from gpu_common import (TOL_E2E, bf16_tensor, check_panels, lib_plan, oracle_layer_step, oracle_mask,
                              rel_l2, within)

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


def _run_steps(tasp, sess, xb, with_logits=False, vocab=0):
    import torch
    S, n, d = xb.shape
    x = bf16_tensor(xb)
    hid = torch.empty((S, n, d), dtype=torch.float32, device="cuda")
    logits = torch.empty((S, n, vocab), dtype=torch.float32, device="cuda") if with_logits else None
    for t in range(S):
        tasp.decode_step(sess if isinstance(sess, list) else [sess], x[t], hid[t],
                         logits[t] if with_logits else None)
    torch.cuda.synchronize()
    return hid.cpu().numpy(), (logits.cpu().numpy() if with_logits else None)


# ------------------------------------------------------------------ single layer (configuration 1)

@pytest.fixture(scope="module")
def layer1(tasp):
    wl = synth.CFG1
    plan = lib_plan(tasp, wl.shape, wl.masks[0])
    yield wl, plan, oracle_mask(wl.shape, wl.masks[0])
    plan.release()


def test_layer1_panels_bit_exact(tasp, layer1):
    wl, plan, mask = layer1
    assert len(mask.keep_groups[0]) == 1 and len(mask.keep_chans[0]) == 832
    check_panels(tasp, plan, wl.shape, mask, 0)
    info = plan.info()
    assert info["launched_flops"] == info["flops_retained"]  # ledger = launched panel shapes
    assert info["flops_retained"] == 655360 + 3072 * 832


def test_layer1_decode_16_steps(tasp, layer1):
    wl, plan, mask = layer1
    sh = wl.shape
    sess = tasp.Session(plan, wl.t_prior + wl.steps)
    sess.fill_synthetic(wl.t_prior, wl.kv_seed)
    xb = synth.step_inputs_bf16(wl.x_seed, wl.steps, 1, sh.d)
    got, _ = _run_steps(tasp, sess, xb)
    assert sess.position == wl.t_prior + wl.steps
    assert sess.device_error() == 0
    ref = forward.decode(sh, mask, synth.bf16_to_f32(xb[:, 0]), wl.t_prior, wl.kv_seed)
    assert within(got[:, 0], ref).all()
    assert rel_l2(got[:, 0], ref) <= TOL_E2E
    sess.release()


def test_layer1_dense_fallback(tasp):
    wl = synth.CFG1
    sh = wl.shape
    plan = tasp.Plan(sh, tasp.all_keep_mask())
    sess = tasp.Session(plan, wl.t_prior + 4)
    sess.fill_synthetic(wl.t_prior, wl.kv_seed)
    xb = synth.step_inputs_bf16(wl.x_seed, 4, 1, sh.d)
    got, _ = _run_steps(tasp, sess, xb)
    ref = forward.decode(sh, maskc.all_keep(sh), synth.bf16_to_f32(xb[:, 0]), wl.t_prior, wl.kv_seed)
    assert within(got[:, 0], ref).all() and rel_l2(got[:, 0], ref) <= TOL_E2E
    sess.release()
    plan.release()


def test_layer1_row_indexed_store_is_bit_identical(tasp, layer1):
    # The paper's one-store check: a plan indexing the shared store and a plan with
    # materialized panels read the same bytes and must give identical outputs.
    wl, plan, _ = layer1
    sh = wl.shape
    plan_z = lib_plan(tasp, sh, wl.masks[0], panel_mode=tasp.PANELS_ROW_INDEXED)
    outs = []
    for p in (plan, plan_z):
        sess = tasp.Session(p, wl.t_prior + 4)
        sess.fill_synthetic(wl.t_prior, wl.kv_seed)
        outs.append(_run_steps(tasp, sess, synth.step_inputs_bf16(wl.x_seed, 4, 1, sh.d))[0])
        sess.release()
    assert np.array_equal(outs[0].view(np.uint32), outs[1].view(np.uint32))
    for item in (tasp.EXPORT_QKV_W, tasp.EXPORT_GU_W, tasp.EXPORT_QKV_S, tasp.EXPORT_GU_S):
        assert np.array_equal(plan.export(0, item), plan_z.export(0, item))
    plan_z.release()


def test_layer1_explicit_ragged_mask(tasp):
    # a mask with a ragged channel count (not a multiple of 16) and both groups kept
    sh = synth.LAYER1
    groups, units = [[0, 1]], [sorted(set(range(0, 1408, 7)))]
    plan = tasp.Plan(sh, tasp.explicit_mask(groups, units))
    mask = maskc.explicit(sh, groups, units)
    assert len(mask.keep_chans[0]) % 16 != 0
    check_panels(tasp, plan, sh, mask, 0)
    sess = tasp.Session(plan, 40)
    sess.fill_synthetic(33, 5)
    xb = synth.step_inputs_bf16(21, 3, 1, sh.d)
    got, _ = _run_steps(tasp, sess, xb)
    ref = forward.decode(sh, mask, synth.bf16_to_f32(xb[:, 0]), 33, 5)
    assert within(got[:, 0], ref).all()
    sess.release()
    plan.release()


def test_layer1_short_context_and_determinism(tasp, layer1):
    # a single prior token (one key before the new one) and two sessions agreeing bit for bit
    wl, plan, mask = layer1
    sh = wl.shape
    outs = []
    for _ in range(2):
        sess = tasp.Session(plan, 8)
        sess.fill_synthetic(1, 99)
        outs.append(_run_steps(tasp, sess, synth.step_inputs_bf16(3, 5, 1, sh.d))[0])
        sess.release()
    assert np.array_equal(outs[0], outs[1])
    ref = forward.decode(sh, mask, synth.bf16_to_f32(synth.step_inputs_bf16(3, 5, 1, sh.d)[:, 0]), 1, 99)
    assert within(outs[0][:, 0], ref).all()


def test_host_buffer_path_equals_device_path(tasp, layer1):
    import torch
    wl, plan, _ = layer1
    sh = wl.shape
    xb = synth.step_inputs_bf16(wl.x_seed, 3, 1, sh.d)
    s1 = tasp.Session(plan, wl.t_prior + 3)
    s1.fill_synthetic(wl.t_prior, wl.kv_seed)
    dev, _ = _run_steps(tasp, s1, xb)
    s2 = tasp.Session(plan, wl.t_prior + 3)
    s2.fill_synthetic(wl.t_prior, wl.kv_seed)
    host = []
    for t in range(3):
        xh = torch.from_numpy(xb[t].view(np.int16)).view(torch.bfloat16).pin_memory()
        hh = torch.empty((1, sh.d), dtype=torch.float32).pin_memory()
        tasp.decode_step_host([s2], xh, hh)
        host.append(hh.numpy().copy())
    assert np.array_equal(np.stack(host), dev)
    s1.release()
    s2.release()


def test_error_codes(tasp, layer1):
    wl, plan, _ = layer1
    sh = wl.shape
    import torch
    other = tasp.Plan(sh, tasp.all_keep_mask())
    a = tasp.Session(plan, 4)
    b = tasp.Session(other, 4)
    x = torch.zeros((2, sh.d), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(tasp.TaspError) as e:
        tasp.decode_step([a, b], x)
    assert e.value.code == tasp.EMASK
    with pytest.raises(tasp.TaspError) as e:
        other.release()  # b still lives on it
    assert e.value.code == tasp.EBUSY
    b.fill_synthetic(4, 1)
    with pytest.raises(tasp.TaspError) as e:
        tasp.decode_step([b], x[:1])
    assert e.value.code == tasp.ECAP
    with pytest.raises(tasp.TaspError) as e:
        tasp.decode_step([a], x[:1], logits=torch.zeros(8, device="cuda"))  # no LM head in this model
    assert e.value.code == tasp.EINVAL
    a.release()
    b.release()
    other.release()


# ------------------------------------------------------------------ Llama-3-8B shape (configuration 2)

@pytest.fixture(scope="module")
def llama8b(tasp):
    wl = synth.CFG2
    plans = [lib_plan(tasp, wl.shape, r) for r in wl.masks]
    masks = [oracle_mask(wl.shape, r) for r in wl.masks]
    yield wl, plans, masks
    for p in plans:
        p.release()


def test_8b_index_lists_all_masks_all_layers(tasp, llama8b):
    wl, plans, masks = llama8b
    for p, m in zip(plans, masks):
        for layer in range(wl.shape.L):
            assert p.export(layer, tasp.EXPORT_KEEP_GROUPS).tolist() == m.keep_groups[layer]
            assert p.export(layer, tasp.EXPORT_KEEP_CHANS).tolist() == m.keep_chans[layer]
        info = p.info()
        assert info["flops_retained"] == m.info["total_flops"] == info["launched_flops"]
        assert info["flops_retained"] / info["flops_dense"] <= 0.57


@pytest.mark.parametrize("mask_id,layer", [(0, 0), (1, 13), (4, 31)])
def test_8b_sampled_layer_panels_and_isolated_layer(tasp, llama8b, mask_id, layer):
    import torch
    wl, plans, masks = llama8b
    sh = wl.shape
    lq = check_panels(tasp, plans[mask_id], sh, masks[mask_id], layer)
    sess = tasp.Session(plans[mask_id], wl.t_prior + 1)
    sess.fill_synthetic(wl.t_prior, wl.kv_seed)
    x = synth.probe_f32(5, layer, sh.d, 4.0)
    xd = torch.from_numpy(x).cuda()
    out = torch.empty_like(xd)
    sess.layer_step(layer, xd, out)
    torch.cuda.synchronize()
    got = out.cpu().numpy()
    ref = oracle_layer_step(sh, masks[mask_id], layer, x, wl.t_prior, wl.kv_seed, lq)
    assert within(got, ref).all(), np.abs(got - ref).max()
    sess.release()


def test_8b_end_to_end_8_steps(tasp, llama8b):
    wl, plans, masks = llama8b
    sh = wl.shape
    steps = 8
    sess = tasp.Session(plans[0], wl.t_prior + steps)
    sess.fill_synthetic(wl.t_prior, wl.kv_seed)
    xb = synth.step_inputs_bf16(wl.x_seed, steps, 1, sh.d)
    got, logits = _run_steps(tasp, sess, xb, with_logits=True, vocab=sh.vocab)
    assert sess.device_error() == 0
    sess.release()
    ref = forward.decode(sh, masks[0], synth.bf16_to_f32(xb[:, 0]), wl.t_prior, wl.kv_seed)
    assert rel_l2(got[:, 0], ref) <= TOL_E2E
    rows = np.arange(0, sh.vocab, 997)
    ref_logits = forward.final_logits(sh, ref, rows=rows)
    assert rel_l2(logits[:, 0, rows], ref_logits) <= TOL_E2E


def test_8b_dense_fallback_isolated_layer(tasp):
    import torch
    wl = synth.CFG2
    sh = wl.shape
    plan = tasp.Plan(sh, tasp.all_keep_mask())
    mask = maskc.all_keep(sh)
    layer = 7
    lq = check_panels(tasp, plan, sh, mask, layer)
    sess = tasp.Session(plan, 600)
    sess.fill_synthetic(512, 3)
    x = synth.probe_f32(9, layer, sh.d, 2.0)
    out = torch.empty(sh.d, dtype=torch.float32, device="cuda")
    sess.layer_step(layer, torch.from_numpy(x).cuda(), out)
    torch.cuda.synchronize()
    ref = oracle_layer_step(sh, mask, layer, x, 512, 3, lq)
    assert within(out.cpu().numpy(), ref).all()
    sess.release()
    plan.release()


# ------------------------------------------------------------------ Llama-3-70B shape (configuration 3)

@pytest.fixture(scope="module")
def llama70b(tasp):
    wl = synth.CFG3
    plan = lib_plan(tasp, wl.shape, wl.masks[0])
    yield wl, plan, oracle_mask(wl.shape, wl.masks[0])
    plan.release()


def test_70b_index_lists_and_ledger(tasp, llama70b):
    wl, plan, mask = llama70b
    for layer in range(wl.shape.L):
        assert plan.export(layer, tasp.EXPORT_KEEP_GROUPS).tolist() == mask.keep_groups[layer]
        assert plan.export(layer, tasp.EXPORT_KEEP_CHANS).tolist() == mask.keep_chans[layer]
    info = plan.info()
    assert info["flops_retained"] == mask.info["total_flops"] == info["launched_flops"]


@pytest.mark.parametrize("layer", [0, 79])
def test_70b_sampled_layer_panels_and_isolated_layer(tasp, llama70b, layer):
    import torch
    wl, plan, mask = llama70b
    sh = wl.shape
    lq = check_panels(tasp, plan, sh, mask, layer)
    sess = tasp.Session(plan, wl.t_prior + wl.steps)
    sess.fill_synthetic(wl.t_prior, wl.kv_seed)
    x = synth.probe_f32(13, layer, sh.d, 8.0)
    out = torch.empty(sh.d, dtype=torch.float32, device="cuda")
    sess.layer_step(layer, torch.from_numpy(x).cuda(), out)
    torch.cuda.synchronize()
    ref = oracle_layer_step(sh, mask, layer, x, wl.t_prior, wl.kv_seed, lq)
    got = out.cpu().numpy()
    assert within(got, ref).all(), np.abs(got - ref).max()
    sess.release()
