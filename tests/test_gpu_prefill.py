"""GPU parity of the prefill path (tcgen05 GEMMs on compacted panels, causal attention over
the kept heads) against the CPU oracle, and of the decode steps that follow it on the same
plan (the mask stays fixed from prefill into decode)."""
import dataclasses

import numpy as np
import pytest

import synth
from oracle import forward
from gpu_common import (TOL_E2E, bf16_tensor, lib_plan, oracle_mask, rel_l2, within)

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


def _prefill_case(tasp, shape, recipe, T, steps, check_layers, logits_rows=None, seed=5):
    import torch
    plan = lib_plan(tasp, shape, recipe)
    mask = oracle_mask(shape, recipe)
    emb = synth.prompt_bf16(seed, 0, T, shape.d)
    logits = torch.empty(shape.vocab, dtype=torch.float32, device="cuda") if shape.vocab else None
    sess = tasp.Session.prefill(plan, bf16_tensor(emb), steps, logits)
    torch.cuda.synchronize()
    assert sess.position == T
    # oracle: causal prefill on the mask-as-zero weights
    Xp, kv = forward.prefill(shape, mask, synth.bf16_to_f32(emb))
    for layer in check_layers:
        kg = mask.keep_groups[layer]
        for which in (0, 1):
            got = synth.bf16_to_f32(sess.kv(layer, which))
            ref = kv[layer][which][kg]
            assert got.shape == ref.shape
            if layer == 0:  # the first layer sees the same input on both sides: per-layer bound
                assert within(got, ref).all(), (layer, which, np.abs(got - ref).max())
            else:  # deeper layers carry the drift of the layers below: end-to-end bound
                assert rel_l2(got, ref) <= TOL_E2E, (layer, which, rel_l2(got, ref))
    if logits is not None:
        rows = logits_rows if logits_rows is not None else np.arange(shape.vocab)
        ref_l = forward.final_logits(shape, Xp[-1:], rows=rows)[0]
        assert rel_l2(logits.cpu().numpy()[rows], ref_l) <= TOL_E2E
    # decode continues on the same plan and cache
    xb = synth.step_inputs_bf16(seed + 1, steps, 1, shape.d)
    x = bf16_tensor(xb)
    hid = torch.empty((steps, 1, shape.d), dtype=torch.float32, device="cuda")
    for t in range(steps):
        tasp.decode_step([sess], x[t], hid[t])
    torch.cuda.synchronize()
    ref = forward.decode(shape, mask, synth.bf16_to_f32(xb[:, 0]), T, 0, prior=lambda l: kv[l])
    got = hid.cpu().numpy()[:, 0]
    assert rel_l2(got, ref) <= TOL_E2E
    assert sess.device_error() == 0
    sess.release()
    plan.release()
    return got, ref


@pytest.mark.parametrize("T", [100, 300])
def test_prefill_single_layer(tasp, T):
    got, ref = _prefill_case(tasp, synth.LAYER1, synth.CFG1.masks[0], T, 4, [0])
    assert within(got, ref).all()


def test_prefill_8b_two_layers_all_masks(tasp):
    sh = dataclasses.replace(synth.LLAMA3_8B, L=2)
    for recipe in synth.CFG4.masks:
        _prefill_case(tasp, sh, recipe, 200, 2, [0, 1], logits_rows=np.arange(0, sh.vocab, 251))


def test_prefill_8b_full_depth_512(tasp):
    sh = synth.LLAMA3_8B
    _prefill_case(tasp, sh, synth.CFG4.masks[0], 512, 2, [0, 15, 31], logits_rows=np.arange(0, sh.vocab, 997))


def test_prefill_8b_two_layers_bench_length(tasp):
    # the benchmark's prompt length (2,048 tokens: two-row-tile GEMMs, 16 query blocks per
    # head in the attention schedule) on a two-layer cut of the 8B widths
    sh = dataclasses.replace(synth.LLAMA3_8B, L=2)
    _prefill_case(tasp, sh, synth.CFG4.masks[0], 2048, 2, [0, 1], logits_rows=np.arange(0, sh.vocab, 499))


def test_prefill_8b_two_layers_longest_prompt(tasp):
    # the longest prompt of the prefill workload (8,192 tokens: 64 query blocks per head in the
    # attention schedule, 64 row tiles per GEMM) on a two-layer cut of the 8B widths
    sh = dataclasses.replace(synth.LLAMA3_8B, L=2)
    _prefill_case(tasp, sh, synth.CFG4.masks[1], 8192, 2, [0, 1], logits_rows=np.arange(0, sh.vocab, 499), seed=9)
