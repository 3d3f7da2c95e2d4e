"""Write the oracle's full-depth Llama-3-70B decode outputs used by tests/test_gpu_full_depth.py.

Calls only ``oracle`` and the seeded generators in ``synth`` (no library code). Six sessions on
the 43% mask of seed 1000, two teacher-forced decode steps each, all 80 layers, weights
regenerated layer by layer (mask-as-zero, FP32):

* session 0: the benchmark's batch-1 decode at context 4,096 (KV seed 7, step inputs of seed 11);
* sessions 1-5: the mixed-turn batch of five at contexts 4,096 / 3,000 / 2,048 / 1,024 / 256
  (KV seeds 7..11, step inputs of seed 16, sessions 0..4 of that stream).

Stored: the residual stream after the last layer [2, 6, 8192] and the logits of every 997th
vocabulary row [2, 6, 129] (final RMSNorm + dense LM head), FP32. About 20 minutes on 8 cores.

    python tests/golden/make_llama70b_full_depth.py
"""
import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import synth  # noqa: E402
from oracle import forward, maskc  # noqa: E402

OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "llama70b_full_depth_decode.npz")
STEPS = 2
T_PRIORS = [4096, 4096, 3000, 2048, 1024, 256]
KV_SEEDS = [7, 7, 8, 9, 10, 11]
LOGIT_STRIDE = 997


def inputs():
    wl = synth.CFG3
    sh = wl.shape
    x_single = synth.step_inputs_bf16(wl.x_seed, STEPS, 1, sh.d)
    x_batch = synth.step_inputs_bf16(wl.x_seed + 5, STEPS, 5, sh.d)
    return np.concatenate([x_single, x_batch], axis=1)  # [STEPS, 6, d] BF16 bits


def main():
    wl = synth.CFG3
    sh = wl.shape
    rec = wl.masks[0]
    sc = synth.mask_scores_u32(rec.mask_seed, sh.L, sh.n_units)
    tg = synth.layer_target_u24(rec.mask_seed, sh.L)
    mask = maskc.compile_mask(sh, sc, tg, rec.budget, rec.r_lo, rec.r_hi)
    xb = inputs()
    t0 = time.time()
    hidden = forward.decode_sessions(sh, mask, synth.bf16_to_f32(xb), T_PRIORS, KV_SEEDS)
    rows = np.arange(0, sh.vocab, LOGIT_STRIDE)
    logits = np.stack([forward.final_logits(sh, hidden[:, i], rows=rows) for i in range(len(T_PRIORS))], axis=1)
    np.savez_compressed(OUT, hidden=hidden.astype(np.float32), logits=logits.astype(np.float32), rows=rows,
                        t_priors=np.array(T_PRIORS), kv_seeds=np.array(KV_SEEDS))
    print(f"wrote {OUT} in {time.time() - t0:.0f} s")


if __name__ == "__main__":
    main()
