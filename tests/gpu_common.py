"""Helpers shared by the GPU parity tests (oracle side + library side set-up)."""
import numpy as np

import synth
from oracle import forward, maskc, pack, weights

TOL_ABS, TOL_REL = 1e-2, 2e-2   # per-layer elementwise bound |gpu - ref| <= 1e-2 + 2e-2 |ref|
TOL_E2E = 3e-2                  # relative L2 on final hidden states


def within(got, ref):
    return np.abs(got - ref) <= TOL_ABS + TOL_REL * np.abs(ref)


def rel_l2(got, ref):
    return float(np.linalg.norm(got - ref) / np.linalg.norm(ref))


def mask_inputs(shape, recipe):
    sc = synth.mask_scores_u32(recipe.mask_seed, shape.L, shape.n_units)
    tg = synth.layer_target_u24(recipe.mask_seed, shape.L)
    return sc, tg


def oracle_mask(shape, recipe):
    sc, tg = mask_inputs(shape, recipe)
    return maskc.compile_mask(shape, sc, tg, recipe.budget, recipe.r_lo, recipe.r_hi)


def lib_plan(tasp, shape, recipe, panel_mode=0):
    sc, tg = mask_inputs(shape, recipe)
    return tasp.Plan(shape, tasp.greedy_mask(sc, tg, recipe.budget, recipe.r_lo, recipe.r_hi, panel_mode))


def bf16_tensor(bits, device="cuda"):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(device)


def check_panels(tasp, plan, shape, mask, layer, lq=None):
    """Index lists and packed INT8 panels + scales of one layer: bit-exact against the oracle."""
    if lq is None:
        lq = weights.gen_layer(shape, layer)
    ref = pack.pack_layer(shape, lq, mask.keep_groups[layer], mask.keep_chans[layer])
    assert plan.export(layer, tasp.EXPORT_KEEP_GROUPS).tolist() == mask.keep_groups[layer]
    assert plan.export(layer, tasp.EXPORT_KEEP_CHANS).tolist() == mask.keep_chans[layer]
    items = {tasp.EXPORT_QKV_W: "qkv_w", tasp.EXPORT_QKV_S: "qkv_s", tasp.EXPORT_O_W: "o_w", tasp.EXPORT_O_S: "o_s",
             tasp.EXPORT_GU_W: "gu_w", tasp.EXPORT_GU_S: "gu_s", tasp.EXPORT_DOWN_W: "down_w",
             tasp.EXPORT_DOWN_S: "down_s"}
    for item, name in items.items():
        got = plan.export(layer, item)
        want = ref[name]
        assert got.shape == want.shape, name
        assert np.array_equal(got.view(np.uint8) if got.dtype == np.int8 else got.view(np.uint32),
                              want.view(np.uint8) if want.dtype == np.int8 else want.view(np.uint32)), name
    return lq


def oracle_layer_step(shape, mask, layer, x, t_prior, kv_seed, lq=None):
    """Oracle output of one layer for input residual x at position t_prior (prior cache only)."""
    if lq is None:
        lq = weights.gen_layer(shape, layer)
    W = weights.dense_zeroed(shape, lq, mask.keep_groups[layer], mask.keep_chans[layer])
    Kc, Vc = forward.prior_cache(shape, layer, kv_seed, t_prior)
    out, _, _ = forward.layer_step(shape, W, x.astype(np.float32), Kc, Vc, t_prior)
    return out
