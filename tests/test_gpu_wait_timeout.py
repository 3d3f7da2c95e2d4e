"""A bounded device wait that runs out: the kernel returns, reports it, and the GPU stays usable.

Every mbarrier wait in the GEMVs gives up after a clock limit, sets bit 0 of the session's
device error word and makes the CTA's later waits return at once. Here the wait is made to run
out without any fault: a test hook shortens the limit to ~1 ms and makes one GEMV launch issue
no weight copies at all, so its consumers' first wait can never complete and no copy is ever
in flight. The test reads the error word back, then decodes normally on the same GPU and
checks the result against the oracle.
"""
import numpy as np
import pytest

import synth
from oracle import forward
from gpu_common import bf16_tensor, lib_plan, oracle_mask, rel_l2, within, TOL_E2E

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


def test_wait_that_runs_out_is_reported_and_gpu_stays_usable(tasp):
    import time
    import torch
    wl = synth.CFG1
    sh = wl.shape
    plan = lib_plan(tasp, sh, wl.masks[0])
    victim = tasp.Session(plan, wl.t_prior + 4)
    victim.fill_synthetic(wl.t_prior, wl.kv_seed)
    assert victim.device_error() == 0
    x = torch.from_numpy(synth.probe_f32(3, 0, sh.d, 2.0)).cuda()
    out = torch.empty_like(x)
    try:
        tasp.test_set_wait_limit(2_000_000)  # ~1 ms of SM clock cycles
        tasp.test_skip_gemv_copies(1)        # the layer's first GEMV (RMSNorm + QKV) streams nothing
        t0 = time.perf_counter()
        victim.layer_step(0, x, out)
        torch.cuda.synchronize()             # the kernel returned on its own
        elapsed = time.perf_counter() - t0
    finally:
        tasp.test_skip_gemv_copies(0)
        tasp.test_set_wait_limit(0)
    assert victim.device_error(clear=True) & 1, "the run-out wait was not reported"
    assert elapsed < 30.0
    # the same session's next layer step runs clean once the word is cleared
    victim.layer_step(0, x, out)
    torch.cuda.synchronize()
    assert victim.device_error() == 0
    victim.release()
    # and a normal decode on the same GPU matches the oracle
    sess = tasp.Session(plan, wl.t_prior + 4)
    sess.fill_synthetic(wl.t_prior, wl.kv_seed)
    xb = synth.step_inputs_bf16(wl.x_seed, 4, 1, sh.d)
    xd = bf16_tensor(xb)
    hid = torch.empty((4, 1, sh.d), dtype=torch.float32, device="cuda")
    for t in range(4):
        tasp.decode_step([sess], xd[t], hid[t])
    torch.cuda.synchronize()
    assert sess.device_error() == 0
    got = hid.cpu().numpy()[:, 0]
    ref = forward.decode(sh, oracle_mask(sh, wl.masks[0]), synth.bf16_to_f32(xb[:, 0]), wl.t_prior, wl.kv_seed)
    assert within(got, ref).all() and rel_l2(got, ref) <= TOL_E2E
    sess.release()
    plan.release()
