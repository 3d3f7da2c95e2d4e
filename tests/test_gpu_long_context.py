"""GPU parity of decode at contexts longer than one attention cluster holds.

Past 16 CTAs x 48 tiles x 16 positions (head dim 64) a kept group's positions are split over
several clusters: each cluster merges its CTAs through distributed shared memory and writes
its partial output and (max, sum) to global scratch, and the last cluster to finish (atomic
ticket) combines them. Covered on the single-layer workload: one session through
tasp_decode_step (16-CTA clusters) and a union step of two plans (8-CTA clusters), against
the oracle.
"""
import numpy as np
import pytest

import synth
from oracle import forward, maskc
from gpu_common import TOL_E2E, bf16_tensor, lib_plan, oracle_mask, rel_l2, within

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


def _decode(tasp, ss, xb, union):
    import torch
    S, n, d = xb.shape
    x = bf16_tensor(xb)
    hid = torch.empty((S, n, d), dtype=torch.float32, device="cuda")
    for t in range(S):
        if union:
            tasp.decode_step_union(ss, x[t], hid[t])
        else:
            tasp.decode_step(ss, x[t], hid[t])
    torch.cuda.synchronize()
    return hid.cpu().numpy()


def test_layer1_decode_beyond_one_cluster(tasp):
    wl = synth.CFG1
    sh = wl.shape
    plan = lib_plan(tasp, sh, wl.masks[0])
    mask = oracle_mask(sh, wl.masks[0])
    tp, steps = 13000, 3  # one 16-CTA cluster holds 12,288 positions at head dim 64
    sess = tasp.Session(plan, tp + steps + 1)
    sess.fill_synthetic(tp, 71)
    xb = synth.step_inputs_bf16(72, steps, 1, sh.d)
    got = _decode(tasp, [sess], xb, False)
    assert sess.device_error() == 0
    sess.release()
    plan.release()
    ref = forward.decode(sh, mask, synth.bf16_to_f32(xb[:, 0]), tp, 71)
    assert within(got[:, 0], ref).all(), np.abs(got[:, 0] - ref).max()
    assert rel_l2(got[:, 0], ref) <= TOL_E2E


def test_union_beyond_one_cluster(tasp):
    wl = synth.CFG1
    sh = wl.shape
    plans = [lib_plan(tasp, sh, wl.masks[0]), tasp.Plan(sh, tasp.all_keep_mask())]
    masks = [oracle_mask(sh, wl.masks[0]), maskc.all_keep(sh)]
    tps, seeds, steps = [7000, 6500], [81, 82], 3  # an 8-CTA cluster holds 6,144 positions
    ss = []
    for pl, tp, sd in zip(plans, tps, seeds):
        s = tasp.Session(pl, tp + steps + 1)
        s.fill_synthetic(tp, sd)
        ss.append(s)
    xb = synth.step_inputs_bf16(83, steps, 2, sh.d)
    got = _decode(tasp, ss, xb, True)
    assert tasp.union_status(ss)[0] == 0
    for s in ss:
        s.release()
    for p in plans:
        p.release()
    for i in range(2):
        ref = forward.decode(sh, masks[i], synth.bf16_to_f32(xb[:, i]), tps[i], seeds[i])
        assert within(got[:, i], ref).all(), (i, np.abs(got[:, i] - ref).max())
        assert rel_l2(got[:, i], ref) <= TOL_E2E


def test_8b_layer_decode_beyond_the_resident_tiles(tasp):
    # head dim 128, 8 clusters of 16 CTAs per kept group: past 8 x 16 x 24 tiles of 16
    # positions each CTA holds more tiles than its shared memory, so it loads them in two
    # batches through the same slots (one 8B layer against the oracle, elementwise)
    import dataclasses
    sh = dataclasses.replace(synth.LLAMA3_8B, L=1, vocab=0)
    recipe = synth.MaskRecipe(1002)
    plan = lib_plan(tasp, sh, recipe)
    mask = oracle_mask(sh, recipe)
    tp, steps = 52000, 2
    sess = tasp.Session(plan, tp + steps)
    sess.fill_synthetic(tp, 91)
    xb = synth.step_inputs_bf16(92, steps, 1, sh.d)
    got = _decode(tasp, [sess], xb, False)
    assert sess.device_error() == 0
    sess.release()
    plan.release()
    ref = forward.decode(sh, mask, synth.bf16_to_f32(xb[:, 0]), tp, 91)
    assert within(got[:, 0], ref).all(), np.abs(got[:, 0] - ref).max()
