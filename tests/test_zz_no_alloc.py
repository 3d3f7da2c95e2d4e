"""The allocation-free decode step against the regular one and the oracle.

tasp_decode_step_static exists for callers that must not enter the CUDA
allocator while decoding (a device-memory budget already handed out, another
library's stream capture in progress, a serving loop that forbids allocator
calls); it takes the attention split scratch from a static device array shared
by every call. Twin sessions (same plan, same prior cache) decode the same inputs
in a row, one through tasp_decode_step and one through the allocation-free call:
their final hidden states (and logits, where the model has an LM head) must agree
within the tolerance of the other parity tests, and with the oracle. The
long-context cases give the sessions a capacity beyond one attention cluster, so
the partial outputs, maxima/sums and merge tickets really go through the static
array, over two calls in a row (the tickets must be back at zero for the second).
Collected last so that a failure here leaves the rest of the suite already run.
"""
import dataclasses

import numpy as np
import pytest

import synth
from oracle import forward
from gpu_common import TOL_ABS, TOL_E2E, TOL_REL, bf16_tensor, lib_plan, oracle_mask, rel_l2, within

pytestmark = pytest.mark.gpu

SHAPE_8B2 = dataclasses.replace(synth.LLAMA3_8B, L=2)


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


def _close(a, b):
    return bool(np.all(np.abs(a - b) <= TOL_ABS + TOL_REL * np.abs(b)))


def _twins(tasp, shape, t_prior, capacity, steps=2, kv_seed=7, x_seed=11):
    """Run `steps` steps on a regular and a static twin; returns (hidden reg, hidden static, logits
    reg, logits static, inputs) as host arrays [steps, ...]."""
    import torch
    plan = lib_plan(tasp, shape, synth.MaskRecipe(1000))
    regular = tasp.Session(plan, capacity)
    static = tasp.Session(plan, capacity)
    for s in (regular, static):
        s.fill_synthetic(t_prior, kv_seed)
    xb = synth.step_inputs_bf16(x_seed, steps, 1, shape.d)
    x = bf16_tensor(xb)
    V = shape.vocab
    h_reg = torch.empty((steps, shape.d), dtype=torch.float32, device="cuda")
    h_sta = torch.empty_like(h_reg)
    l_reg = torch.empty((steps, V), dtype=torch.float32, device="cuda") if V else None
    l_sta = torch.empty_like(l_reg) if V else None
    for t in range(steps):  # calls in a row
        tasp.decode_step([regular], x[t], h_reg[t:t + 1], l_reg[t:t + 1] if V else None)
        tasp.decode_step_static(static, x[t], h_sta[t:t + 1], l_sta[t:t + 1] if V else None)
    torch.cuda.synchronize()
    assert static.position == regular.position == t_prior + steps
    assert static.device_error() == 0 and regular.device_error() == 0
    out = (h_reg.cpu().numpy(), h_sta.cpu().numpy(), l_reg.cpu().numpy() if V else None,
           l_sta.cpu().numpy() if V else None, xb)
    regular.release()
    static.release()
    plan.release()
    return out


@pytest.mark.parametrize("shape,t_prior", [(synth.LAYER1, 128), (SHAPE_8B2, 700)])
def test_static_step_matches_regular_step(tasp, shape, t_prior):
    h_reg, h_sta, l_reg, l_sta, _ = _twins(tasp, shape, t_prior, t_prior + 2)
    assert _close(h_sta, h_reg)
    if shape.vocab:
        assert _close(l_sta, l_reg)


@pytest.mark.parametrize("shape,t_prior,capacity", [
    (synth.LAYER1, 13000, 13010),  # head dim 64: one 16-CTA cluster reaches 12,288 positions -> 2 clusters
    (SHAPE_8B2, 6500, 13000),      # head dim 128: one cluster reaches 6,144 positions -> 3 clusters
])
def test_static_step_beyond_one_cluster_matches_regular_and_oracle(tasp, shape, t_prior, capacity):
    h_reg, h_sta, l_reg, l_sta, xb = _twins(tasp, shape, t_prior, capacity, kv_seed=31, x_seed=32)
    assert _close(h_sta, h_reg)
    if shape.vocab:
        assert _close(l_sta, l_reg)
    mask = oracle_mask(shape, synth.MaskRecipe(1000))
    ref = forward.decode(shape, mask, synth.bf16_to_f32(xb[:, 0]), t_prior, 31)
    assert rel_l2(h_sta, ref) <= TOL_E2E
    if shape.L == 1:
        assert within(h_sta, ref).all(), np.abs(h_sta - ref).max()


def test_static_step_allocates_nothing(tasp):
    import torch
    shape = SHAPE_8B2
    plan = lib_plan(tasp, shape, synth.MaskRecipe(1000))
    sess = tasp.Session(plan, 13000)  # several attention clusters: the static array is in use
    sess.fill_synthetic(6500, 5)
    x = bf16_tensor(synth.step_inputs_bf16(6, 4, 1, shape.d))
    hid = torch.empty((4, shape.d), dtype=torch.float32, device="cuda")
    logits = torch.empty((4, shape.vocab), dtype=torch.float32, device="cuda")
    tasp.decode_step_static(sess, x[0], hid[0:1], logits[0:1])  # first call: address lookup, kernel loading
    torch.cuda.synchronize()
    lib0, torch0, free0 = tasp.memory_in_use(), torch.cuda.memory_allocated(), torch.cuda.mem_get_info()[0]
    for t in range(1, 4):
        tasp.decode_step_static(sess, x[t], hid[t:t + 1], logits[t:t + 1])
    torch.cuda.synchronize()
    assert tasp.memory_in_use() == lib0
    assert torch.cuda.memory_allocated() == torch0
    assert torch.cuda.mem_get_info()[0] == free0
    assert sess.position == 6504 and sess.device_error() == 0
    sess.release()
    plan.release()


def test_static_step_refuses_a_plan_beyond_the_array(tasp):
    import torch
    # 16 KV heads of one query head each, all kept: 16 groups in a layer, more than the array takes
    shape = synth.ModelShape(L=1, d=256, Hq=16, Hkv=16, dh=64, df=256, vocab=0, chan_unit=16, seed=5)
    plan = tasp.Plan(shape, tasp.all_keep_mask())
    sess = tasp.Session(plan, 64)
    sess.fill_synthetic(16, 3)
    x = bf16_tensor(synth.step_inputs_bf16(4, 1, 1, shape.d))
    hid = torch.empty((1, shape.d), dtype=torch.float32, device="cuda")
    with pytest.raises(tasp.TaspError) as ei:
        tasp.decode_step_static(sess, x[0], hid)
    assert ei.value.code == tasp.EINVAL
    assert sess.position == 16
    # the regular step takes the same plan
    tasp.decode_step([sess], x[0], hid)
    torch.cuda.synchronize()
    assert sess.position == 17 and sess.device_error() == 0
    sess.release()
    plan.release()
