"""GPU parity of batched decode: several sessions of one plan in one step.

The GEMVs of a step read each weight byte once for up to four sessions and one
attention grid covers them, each session on its own KV cache and position (turns
that share a mask are decoded together). Every session must match the oracle's
decode of that session alone, and the batch must agree with single-session steps
up to FP32 summation order. Groups of 2 and 4 vectors, K passes (rows longer than
the register-resident slice of a 4-vector pass) and the 4 + 1 split of five sessions
are all covered.
"""
import numpy as np
import pytest

import synth
from oracle import forward
from gpu_common import TOL_E2E, bf16_tensor, lib_plan, oracle_mask, rel_l2, within

pytestmark = pytest.mark.gpu

# Relative L2 between a batched and a single-session run. The two sum the projections in
# different FP32 orders (other rows per stage, K passes, cross-warp order); where a new key
# or value lands next to a BF16 rounding boundary of the KV cache the two caches then hold
# neighbouring BF16 values (2^-8 apart), which attention carries into later outputs. A
# wrong session, row or position would differ at O(0.1-1).
TOL_BATCH = 1e-3


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


def _cap(tp, extra, i):
    return tp + extra + 5 * i  # capacities (KV row strides) differ between sessions


def _sessions(tasp, plan, t_priors, kv_seeds, extra):
    out = []
    for i, (tp, ks) in enumerate(zip(t_priors, kv_seeds)):
        s = tasp.Session(plan, _cap(tp, extra, i))
        s.fill_synthetic(tp, ks)
        out.append(s)
    return out


def _run(tasp, sessions, xb, vocab=0):
    """xb [S, n, d] BF16 bits; returns hidden [S, n, d] (and logits [S, n, V])."""
    import torch
    S, n, d = xb.shape
    x = bf16_tensor(xb)
    hid = torch.empty((S, n, d), dtype=torch.float32, device="cuda")
    lg = torch.empty((S, n, vocab), dtype=torch.float32, device="cuda") if vocab else None
    for t in range(S):
        tasp.decode_step(sessions, x[t], hid[t], lg[t] if vocab else None)
    torch.cuda.synchronize()
    return hid.cpu().numpy(), (lg.cpu().numpy() if vocab else None)


def _singles(tasp, plan, t_priors, kv_seeds, xb, vocab=0):
    hs, ls = [], []
    for i, (tp, ks) in enumerate(zip(t_priors, kv_seeds)):
        s = tasp.Session(plan, _cap(tp, xb.shape[0], i))
        s.fill_synthetic(tp, ks)
        h, l = _run(tasp, [s], xb[:, i:i + 1], vocab)
        assert s.device_error() == 0
        s.release()
        hs.append(h[:, 0])
        ls.append(l[:, 0] if vocab else None)
    return hs, ls


# ------------------------------------------------------------------ single layer

@pytest.fixture(scope="module")
def layer1(tasp):
    wl = synth.CFG1
    plan = lib_plan(tasp, wl.shape, wl.masks[0])
    yield wl, plan, oracle_mask(wl.shape, wl.masks[0])
    plan.release()


@pytest.mark.parametrize("n", [2, 3, 4, 5])
def test_layer1_batch_matches_oracle_and_single(tasp, layer1, n):
    wl, plan, mask = layer1
    sh = wl.shape
    steps = 6
    t_priors = [128, 70, 100, 17, 1][:n]        # ragged contexts, one nearly empty
    kv_seeds = [wl.kv_seed + i for i in range(n)]
    xb = synth.step_inputs_bf16(wl.x_seed + n, steps, n, sh.d)
    ss = _sessions(tasp, plan, t_priors, kv_seeds, steps)
    got, _ = _run(tasp, ss, xb)
    for i, s in enumerate(ss):
        assert s.position == t_priors[i] + steps
        assert s.device_error() == 0
    ref = forward.decode_sessions(sh, mask, synth.bf16_to_f32(xb), t_priors, kv_seeds)
    for i in range(n):
        assert within(got[:, i], ref[:, i]).all(), (i, np.abs(got[:, i] - ref[:, i]).max())
        assert rel_l2(got[:, i], ref[:, i]) <= TOL_E2E
    singles, _ = _singles(tasp, plan, t_priors, kv_seeds, xb)
    for i in range(n):
        assert rel_l2(got[:, i], singles[i]) <= TOL_BATCH
    for s in ss:
        s.release()


def test_layer1_batch_host_path_equals_device_path(tasp, layer1):
    import torch
    wl, plan, _ = layer1
    sh = wl.shape
    n, steps = 3, 3
    t_priors, kv_seeds = [128, 40, 77], [1, 2, 3]
    xb = synth.step_inputs_bf16(17, steps, n, sh.d)
    ss = _sessions(tasp, plan, t_priors, kv_seeds, steps)
    dev, _ = _run(tasp, ss, xb)
    for s in ss:
        s.release()
    ss = _sessions(tasp, plan, t_priors, kv_seeds, steps)
    host = np.empty((steps, n, sh.d), np.float32)
    for t in range(steps):
        x = torch.from_numpy(xb[t].view(np.int16)).view(torch.bfloat16).pin_memory()
        h = torch.empty((n, sh.d), dtype=torch.float32).pin_memory()
        tasp.decode_step_host(ss, x, h)
        host[t] = h.numpy()
    assert np.array_equal(dev.view(np.uint32), host.view(np.uint32))
    for s in ss:
        s.release()


def test_batch_errors_and_release(tasp, layer1):
    wl, plan, _ = layer1
    sh = wl.shape
    import torch
    other = lib_plan(tasp, sh, wl.masks[0])
    a, b = _sessions(tasp, plan, [10, 10], [1, 2], 4)
    (c,) = _sessions(tasp, other, [10], [1], 4)
    x = bf16_tensor(synth.step_inputs_bf16(3, 1, 3, sh.d)[0])
    with pytest.raises(tasp.TaspError) as e:
        tasp.decode_step([a, b, c], x)
    assert e.value.code == tasp.EMASK                     # one plan per step: no KV reuse across masks
    with pytest.raises(tasp.TaspError) as e:
        tasp.decode_step([a, a], x[:2])
    assert e.value.code == tasp.EINVAL
    with pytest.raises(ValueError):
        tasp.decode_step([a, b], x[:1])                   # input buffer too small for two sessions
    # a batch survives repeated steps, and releasing one session drops its batch
    tasp.decode_step([a, b], x[:2])
    tasp.decode_step([a, b], x[:2])
    b.release()
    tasp.decode_step([a], x[:1])
    torch.cuda.synchronize()
    assert a.position == 13 and a.device_error() == 0
    a.release()
    c.release()
    other.release()


# ------------------------------------------------------------------ Llama-3-8B / 70B widths
# Through many layers of random weights a perturbation grows by ~1.2x per layer, so the
# tight batch-versus-single comparisons run on two-layer cuts of the full widths (the
# same kernels, the same K passes); full-depth runs are checked against the oracle.

def _cut(shape, L):
    import dataclasses
    return dataclasses.replace(shape, L=L)


@pytest.mark.parametrize("cfg,n", [(2, 4), (3, 5)])
def test_full_width_two_layer_batch_matches_oracle_and_single(tasp, cfg, n):
    # 8B width, 4 sessions: the down projection (up to 14,336 kept channels) takes two K
    # passes of a 4-vector kernel; 70B width, 4 + 1 sessions: up to four passes, and
    # the LM head's two passes
    wl = synth.CONFIGS[cfg]
    sh = _cut(wl.shape, 2)
    recipe = wl.masks[0]
    plan = lib_plan(tasp, sh, recipe)
    mask = oracle_mask(sh, recipe)
    steps = 2
    t_priors = [wl.t_prior, 1000, 517, 3, 256][:n]
    kv_seeds = [wl.kv_seed + i for i in range(n)]
    xb = synth.step_inputs_bf16(wl.x_seed + n, steps, n, sh.d)
    ss = _sessions(tasp, plan, t_priors, kv_seeds, steps)
    got, logits = _run(tasp, ss, xb, sh.vocab)
    for s in ss:
        assert s.device_error() == 0
        s.release()
    ref = forward.decode_sessions(sh, mask, synth.bf16_to_f32(xb), t_priors, kv_seeds)
    rows = np.arange(0, sh.vocab, 4999)
    for i in range(n):
        # two layers deep: the relative-L2 bound (the elementwise one is for isolated layers)
        assert rel_l2(got[:, i], ref[:, i]) <= TOL_E2E, i
        ref_l = forward.final_logits(sh, ref[:, i], rows=rows)
        assert rel_l2(logits[:, i, rows], ref_l) <= TOL_E2E, i
    singles, single_logits = _singles(tasp, plan, t_priors, kv_seeds, xb, sh.vocab)
    for i in range(n):
        assert rel_l2(got[:, i], singles[i]) <= TOL_BATCH, i
        assert rel_l2(logits[:, i], single_logits[i]) <= TOL_BATCH, i
    plan.release()


def test_8b_batch_of_four_end_to_end(tasp):
    wl = synth.CFG2
    sh = wl.shape
    plan = lib_plan(tasp, sh, wl.masks[1])
    mask = oracle_mask(sh, wl.masks[1])
    n, steps = 4, 3
    t_priors = [2048, 1000, 517, 3]
    kv_seeds = [wl.kv_seed, 11, 12, 13]
    xb = synth.step_inputs_bf16(wl.x_seed + 4, steps, n, sh.d)
    ss = _sessions(tasp, plan, t_priors, kv_seeds, steps)
    got, logits = _run(tasp, ss, xb, sh.vocab)
    for s in ss:
        assert s.device_error() == 0
        s.release()
    ref = forward.decode_sessions(sh, mask, synth.bf16_to_f32(xb), t_priors, kv_seeds)
    rows = np.arange(0, sh.vocab, 997)
    singles, _ = _singles(tasp, plan, t_priors, kv_seeds, xb)
    for i in range(n):
        err = rel_l2(got[:, i], ref[:, i])
        assert err <= TOL_E2E, i
        assert rel_l2(logits[:, i, rows], forward.final_logits(sh, ref[:, i], rows=rows)) <= TOL_E2E, i
        # 32 layers deep the BF16 rounding noise of the KV cache is of the order of the
        # distance to the (FP32-cache) oracle, ~5e-4
        assert rel_l2(got[:, i], singles[i]) <= 2 * TOL_BATCH, i
    plan.release()


def test_70b_width_row_indexed_batch_is_bit_identical(tasp):
    # the mixed-turn bench's configuration: a group of four sessions on a plan whose Q/K/V and
    # gate/up panels are row maps into the shared store reads the same bytes as materialized
    # panels, so every output bit agrees (the paper's one-store check, at 70B widths)
    wl = synth.CFG5
    sh = _cut(wl.shape, 2)
    recipe = wl.masks[2]
    n, steps = 4, 2
    t_priors = [1500, 700, 256, 2000]
    kv_seeds = [wl.kv_seed + i for i in range(n)]
    xb = synth.step_inputs_bf16(wl.x_seed, steps, n, sh.d)
    outs = []
    for mode in (tasp.PANELS_COMPACT, tasp.PANELS_ROW_INDEXED):
        plan = lib_plan(tasp, sh, recipe, panel_mode=mode)
        ss = _sessions(tasp, plan, t_priors, kv_seeds, steps)
        outs.append(_run(tasp, ss, xb, sh.vocab))
        for s in ss:
            assert s.device_error() == 0
            s.release()
        plan.release()
    (h0, l0), (h1, l1) = outs
    assert np.array_equal(h0.view(np.uint32), h1.view(np.uint32))
    assert np.array_equal(l0.view(np.uint32), l1.view(np.uint32))
