"""GPU parity of query-head-granular masks (Sec. 3.3: query-head candidates, a KV head kept
whenever one of its heads is) against the oracle, through the C ABI: panels and kept lists
bit-exact, decode and prefill elementwise, compact = row-indexed panels bit for bit, and the
union step refusing plans with partial groups."""
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
    sh = dataclasses.replace(synth.LLAMA3_8B, L=2)
    seed = 1000
    sc = synth.mask_scores_u32(seed, sh.L, sh.Hq + sh.n_chan_units)
    tg = synth.layer_target_u24(seed, sh.L)
    mask = maskc.compile_mask_qheads(sh, sc, tg, 0.4, 0.2, 0.6)
    plan = tasp.Plan(sh, tasp.greedy_qhead_mask(sc, tg, 0.4, 0.2, 0.6))
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


def test_union_refuses_partial_groups(tasp):
    import torch
    sh = dataclasses.replace(synth.LLAMA3_8B, L=1)
    plan = tasp.Plan(sh, tasp.explicit_qhead_mask([[0, 1, 2, 8]], [[0, 3]]))
    sess = tasp.Session(plan, 8)
    sess.fill_synthetic(4, 1)
    x = torch.zeros((1, sh.d), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(tasp.TaspError) as e:
        tasp.decode_step_union([sess], x)
    assert e.value.code == tasp.EUNSUP
    sess.release()
    plan.release()


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
