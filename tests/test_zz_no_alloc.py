"""The allocation-free decode step against the regular one.

tasp_decode_step_static exists for callers that must not enter the CUDA
allocator while decoding; it takes the attention split scratch from a static
device array shared by every call. Here two twin sessions (same plan, same
prior cache) decode the same two inputs in a row, one through tasp_decode_step
and one through the allocation-free call, and their final hidden states (and
logits, where the model has an LM head) must agree within the tolerance of the
other parity tests. Collected last so that a failure here leaves the rest of the
suite already run.
"""
import dataclasses

import numpy as np
import pytest

import synth
from gpu_common import TOL_ABS, TOL_REL, bf16_tensor, lib_plan

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


def _close(a, b):
    return bool(np.all(np.abs(a - b) <= TOL_ABS + TOL_REL * np.abs(b)))


@pytest.mark.parametrize("shape,t_prior", [(synth.LAYER1, 128), (dataclasses.replace(synth.LLAMA3_8B, L=2), 700)])
def test_static_step_matches_regular_step(tasp, shape, t_prior):
    import torch
    plan = lib_plan(tasp, shape, synth.MaskRecipe(1000))
    steps = 2
    regular = tasp.Session(plan, t_prior + steps)
    static = tasp.Session(plan, t_prior + steps)
    for s in (regular, static):
        s.fill_synthetic(t_prior, 7)
    x = bf16_tensor(synth.step_inputs_bf16(11, steps, 1, shape.d))
    V = shape.vocab
    for t in range(steps):  # two calls in a row
        h_reg = torch.empty((1, shape.d), dtype=torch.float32, device="cuda")
        h_sta = torch.empty_like(h_reg)
        l_reg = torch.empty((1, V), dtype=torch.float32, device="cuda") if V else None
        l_sta = torch.empty_like(l_reg) if V else None
        tasp.decode_step([regular], x[t], h_reg, l_reg)
        tasp.decode_step_static(static, x[t], h_sta, l_sta)
        torch.cuda.synchronize()
        assert _close(h_sta.cpu().numpy(), h_reg.cpu().numpy())
        if V:
            assert _close(l_sta.cpu().numpy(), l_reg.cpu().numpy())
    assert static.position == regular.position == t_prior + steps
    assert static.device_error() == 0 and regular.device_error() == 0
    regular.release()
    static.release()
    plan.release()
