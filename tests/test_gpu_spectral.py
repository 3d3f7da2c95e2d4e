"""GPU spectral descriptors of the candidate units against the oracle (Sec. 3.1, Eqs. 1-4;
Appendix "Exact candidate feature construction").

The device builds each candidate's block from the synthetic weights rounded to BF16 (the
checkpoint precision the paper reads), forms its Gram matrix on the tensor cores (FP16 operands
holding the BF16 values, FP32 accumulation) and takes the eigenvalues in FP32 with a symmetric
eigensolver; the oracle takes the singular values of the same BF16-rounded block in FP64.

Tolerances, from the arithmetic: each Gram entry sums d products in FP32, a relative error of
order sqrt(d) 2^-24 of the entries' scale (~5e-6 at d = 8192), and an FP32 eigensolver adds
n 2^-24 lambda_max at most; the eigenvalues are compared to 2e-4 lambda_max. The effective rank,
SETOL and the spectral norm are smooth in them (relative 1e-4, absolute 1e-4, relative 1e-4). The
tail cut lambda_min is an argmin over ~n candidates: where both sides pick the same eigenvalue
(rank), alpha and the KS distance agree to 1e-3 relative; where they pick different ones, the
oracle's own KS distance at the device's pick must be within 2e-3 of its optimum (a near-tie that
rounding may break either way).
"""
import dataclasses

import numpy as np
import pytest

import synth
from oracle import spectral

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


def _bf16_weights(shape, layer):
    W = spectral.dense_f32(shape, layer)
    return {k: synth.bf16_to_f32(synth.bf16_bits(v)) for k, v in W.items()}


def _check(shape, layer, feat, lam, idx, W):
    names = ("alpha", "r_eff", "spectral_norm", "setol", "lambda_min", "ks")
    for i in idx:
        head = i < shape.Hq
        block = spectral.head_block(shape, W, i) if head else spectral.channel_block(shape, W, i - shape.Hq)
        ref_lam = spectral.eigenvalues(block, shape.d)
        got_lam = lam[i]
        assert got_lam.shape == ref_lam.shape
        assert np.max(np.abs(got_lam - ref_lam)) <= 2e-4 * ref_lam[0], (i, np.max(np.abs(got_lam - ref_lam)) / ref_lam[0])
        ref = spectral.features(block, shape.d, layer, shape.L, head)
        got = dict(zip(names, feat[i]))
        assert abs(got["r_eff"] - ref.r_eff) <= 1e-4 * ref.r_eff, (i, got["r_eff"], ref.r_eff)
        assert abs(got["spectral_norm"] - ref.spectral_norm) <= 1e-4 * ref.spectral_norm, i
        k_got = int(np.argmin(np.abs(ref_lam - got["lambda_min"])))  # the device's pick as a rank
        k_ref = int(np.argmin(np.abs(ref_lam - ref.lam_min)))
        if k_got == k_ref:
            assert abs(got["alpha"] - ref.alpha) <= 1e-3 * ref.alpha, (i, got["alpha"], ref.alpha)
            assert abs(got["ks"] - ref.ks) <= 1e-3 * max(ref.ks, 1e-3), (i, got["ks"], ref.ks)
            assert abs(got["setol"] - ref.setol) <= 1e-4, (i, got["setol"], ref.setol)
        else:  # a near-tie of the KS distance: the device's cut is optimal within rounding
            x = ref_lam[k_got]
            D_at = spectral.ks_distance(ref_lam, x, spectral.tail_alpha(ref_lam, x))
            assert D_at - ref.ks <= 2e-3, (i, D_at, ref.ks)
        assert 0.0 < got["setol"] <= 1.0 and got["alpha"] > 0.0


def test_spectral_small_shape_all_candidates(tasp):
    # 8 heads of [256, 1024] blocks and 3 channel groups of [768, 1024]
    sh = synth.ModelShape(L=2, d=1024, Hq=8, Hkv=2, dh=64, df=768, vocab=0, chan_unit=256, seed=3)
    layer = 1
    feat, lam = tasp.spectral_layer(sh, layer)
    assert feat.shape == (sh.Hq + sh.df // sh.chan_unit, 6) and np.isfinite(feat).all()
    _check(sh, layer, feat, lam, range(len(lam)), _bf16_weights(sh, layer))


def test_spectral_8b_layer_sampled_candidates(tasp):
    # the 8B widths: heads [512, 4096], channel groups [3072, 4096]; the device computes all 46
    # candidates of the layer, the oracle checks a sample of both kinds
    sh = dataclasses.replace(synth.LLAMA3_8B, L=4)
    layer = 2
    feat, lam = tasp.spectral_layer(sh, layer)
    assert np.isfinite(feat).all()
    _check(sh, layer, feat, lam, [0, 13, 31, sh.Hq + 0, sh.Hq + 9], _bf16_weights(sh, layer))
    # every head's block is i.i.d. Gaussian: its spectrum lies near the Marchenko-Pastur support
    q = 4 * sh.dh / sh.d
    s2 = synth.WEIGHT_SIGMA ** 2
    lo, hi = s2 * (1 - np.sqrt(q)) ** 2, s2 * (1 + np.sqrt(q)) ** 2
    for i in range(sh.Hq):
        assert lam[i][0] <= 1.1 * hi and lam[i][-1] >= 0.9 * lo, i


def test_spectral_refuses_tall_blocks(tasp):
    sh = synth.ModelShape(L=1, d=128, Hq=4, Hkv=2, dh=64, df=256, vocab=0, chan_unit=64, seed=3)
    with pytest.raises(tasp.TaspError) as ei:
        tasp.spectral_layer(sh, 0)
    assert ei.value.code == tasp.EUNSUP
