"""Full-depth Llama-3-70B decode against the oracle (the benchmark's configuration).

All 80 layers of the 43% mask, two teacher-forced steps with logits, compared on the final
hidden state (relative L2 <= 3e-2) and on every 997th logit row:

* one session at context 4,096 through the one-session kernels, graph-replayed (the
  benchmark's batch-1 decode);
* five sessions at contexts 4,096 / 3,000 / 2,048 / 1,024 / 256 in one call (a group of four
  through the batched GEMVs plus one through the one-session kernels: the mixed-turn batch).

The oracle's outputs (mask-as-zero FP32 decode, weights regenerated layer by layer) take
about 20 CPU minutes, so they are stored in tests/golden/llama70b_full_depth_decode.npz by
tests/golden/make_llama70b_full_depth.py, which calls only the oracle and the generators.
"""
import os

import numpy as np
import pytest

import synth
from gpu_common import TOL_E2E, bf16_tensor, lib_plan, rel_l2

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "llama70b_full_depth_decode.npz")


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


def _load_golden():
    import importlib.util
    spec = importlib.util.spec_from_file_location(
        "make_llama70b_full_depth", os.path.join(os.path.dirname(GOLDEN), "make_llama70b_full_depth.py"))
    mk = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mk)
    g = np.load(GOLDEN)
    assert g["t_priors"].tolist() == mk.T_PRIORS and g["kv_seeds"].tolist() == mk.KV_SEEDS
    return mk, g


def _run(tasp, sessions, xb, vocab):
    import torch
    S, n, d = xb.shape
    x = bf16_tensor(xb)
    hid = torch.empty((S, n, d), dtype=torch.float32, device="cuda")
    lg = torch.empty((S, n, vocab), dtype=torch.float32, device="cuda")
    for t in range(S):
        tasp.decode_step(sessions, x[t], hid[t], lg[t])
    torch.cuda.synchronize()
    return hid.cpu().numpy(), lg.cpu().numpy()


def test_llama70b_full_depth_decode_matches_oracle(tasp):
    mk, g = _load_golden()
    wl = synth.CFG3
    sh = wl.shape
    xb = mk.inputs()
    steps = xb.shape[0]
    plan = lib_plan(tasp, sh, wl.masks[0])
    ss = []
    for i, (tp, ks) in enumerate(zip(mk.T_PRIORS, mk.KV_SEEDS)):
        s = tasp.Session(plan, tp + steps + 3 * i)  # capacities (KV row strides) differ
        s.fill_synthetic(tp, ks)
        ss.append(s)
    h1, l1 = _run(tasp, ss[:1], xb[:, :1], sh.vocab)  # batch 1, the benchmark's step
    h5, l5 = _run(tasp, ss[1:], xb[:, 1:], sh.vocab)  # five sessions in one call (4 + 1)
    for i, s in enumerate(ss):
        assert s.device_error() == 0
        assert s.position == mk.T_PRIORS[i] + steps
        s.release()
    plan.release()
    hid = np.concatenate([h1, h5], axis=1)
    lg = np.concatenate([l1, l5], axis=1)[:, :, g["rows"]]
    assert np.isfinite(hid).all() and np.isfinite(lg).all()
    for i in range(len(mk.T_PRIORS)):
        e_h = rel_l2(hid[:, i], g["hidden"][:, i])
        e_l = rel_l2(lg[:, i], g["logits"][:, i])
        assert e_h <= TOL_E2E, (i, e_h)
        assert e_l <= TOL_E2E, (i, e_l)
