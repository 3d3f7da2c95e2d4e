"""Pins of the oracle's spectral descriptors (Sec. 3.1: Pareto tail exponent with a
KS-selected cutoff, SETOL, effective rank, spectral norm; Appendix, Eq. candidate-features:
the stacked blocks of attention heads and SwiGLU channel groups)."""
import numpy as np
import pytest
import scipy.stats

import synth
from oracle import spectral as sp


def _with_singular_values(s, rows, cols, seed=0):
    rng = np.random.default_rng(seed)
    U, _ = np.linalg.qr(rng.standard_normal((rows, rows)))
    V, _ = np.linalg.qr(rng.standard_normal((cols, cols)))
    S = np.zeros((rows, cols))
    S[np.arange(len(s)), np.arange(len(s))] = s
    return U @ S @ V.T


def test_effective_rank_closed_forms():
    assert sp.effective_rank(np.full(37, 0.25)) == pytest.approx(37.0, rel=1e-13)
    assert sp.effective_rank(np.array([3.0, 0.0, 0.0])) == pytest.approx(1.0, rel=1e-15)
    # two eigenvalues in ratio 3:1: exp(-(3/4 log 3/4 + 1/4 log 1/4))
    want = np.exp(-(0.75 * np.log(0.75) + 0.25 * np.log(0.25)))
    assert sp.effective_rank(np.array([3.0, 1.0])) == pytest.approx(want, rel=1e-14)


def test_spectral_norm_and_eigenvalues_from_known_singular_values():
    s = np.array([5.0, 3.0, 2.5, 1.0, 0.5, 0.25])
    W = _with_singular_values(s, 6, 40)
    lam = sp.eigenvalues(W, 40)
    assert np.allclose(lam, s * s / 40, rtol=1e-12)
    f = sp.features(W, 40, 0, 1, True)
    assert f.spectral_norm == pytest.approx(5.0, rel=1e-12)
    rng = np.random.default_rng(4)
    A = rng.standard_normal((30, 70))
    assert sp.features(A, 70, 0, 1, False).spectral_norm == pytest.approx(np.linalg.norm(A, 2), rel=1e-12)


def _pareto_sample(n, alpha, lam_min, seed=1):
    # stratified quantiles of P(lambda > x) = (x / lam_min)^-alpha
    u = (np.arange(n) + 0.5) / n
    return lam_min * (1.0 - u) ** (-1.0 / alpha)


def test_alpha_is_the_pareto_maximum_likelihood_estimate():
    rng = np.random.default_rng(2)
    x = 0.3 * (1 + rng.pareto(1.7, 400))
    a = sp.tail_alpha(x, 0.3)
    b, loc, scale = scipy.stats.pareto.fit(x, floc=0, fscale=0.3)
    assert a == pytest.approx(b, rel=1e-9)
    # a stratified sample of an exact Pareto law recovers its exponent
    assert sp.tail_alpha(_pareto_sample(20000, 2.5, 1.0), 1.0) == pytest.approx(2.5, rel=2e-3)


def test_ks_distance_matches_scipy():
    rng = np.random.default_rng(3)
    lam = np.concatenate([rng.uniform(0, 1, 300), 1.0 * (1 + rng.pareto(2.0, 120))])
    for lam_min in (0.5, 1.0, 1.7):
        a = sp.tail_alpha(lam, lam_min)
        tail = lam[lam >= lam_min]
        ref = scipy.stats.kstest(tail, lambda t: 1.0 - (t / lam_min) ** (-a)).statistic
        assert sp.ks_distance(lam, lam_min, a) == pytest.approx(ref, rel=1e-12, abs=1e-15)


def test_cutoff_is_the_ks_minimizer():
    # brute force over every admissible cutoff with scipy's KS statistic
    rng = np.random.default_rng(5)
    lam = np.concatenate([rng.uniform(0.1, 2.0, 200), 2.0 * (1 + rng.pareto(2.0, 80))])
    lam_min, a, D = sp.fit_tail(lam)
    vals = np.unique(lam)[:-1]
    Ds = []
    for x in vals:
        ax = len(lam[lam >= x]) / np.sum(np.log(lam[lam >= x] / x))
        Ds.append(scipy.stats.kstest(lam[lam >= x], lambda t, x=x, ax=ax: 1.0 - (t / x) ** (-ax)).statistic)
    k = int(np.argmin(Ds))
    assert lam_min == vals[k] and D == pytest.approx(Ds[k], rel=1e-12)
    # the mixture's Pareto part starts at 2 with exponent 2
    assert 1.8 <= lam_min <= 2.6 and 1.5 <= a <= 2.6


def test_setol_hand_cases_and_scale_invariance():
    lam = np.array([8.0, 4.0, 2.0, 1.0, 1.0])
    assert sp.setol(lam, 1.0) == 1.0
    assert sp.setol(lam, 4.0) == pytest.approx(12.0 / 16.0)
    rng = np.random.default_rng(6)
    W = rng.standard_normal((24, 96)) * np.linspace(0.2, 3.0, 96)
    f1, f2 = sp.features(W, 96, 2, 5, True), sp.features(-7.5 * W, 96, 2, 5, True)
    assert f2.alpha == pytest.approx(f1.alpha, rel=1e-9)
    assert f2.setol == pytest.approx(f1.setol, rel=1e-12)
    assert f2.r_eff == pytest.approx(f1.r_eff, rel=1e-12)
    assert f2.spectral_norm == pytest.approx(7.5 * f1.spectral_norm, rel=1e-12)
    assert f1.layer_pos == 0.5 and f1.is_attention


def test_candidate_blocks_come_from_their_projections():
    sh = synth.tiny_shape(L=1, chan_unit=16)
    W = sp.dense_f32(sh, 0)
    h = 2  # group h // g = 1 (g = 2); a map h % H_kv would give group 0
    B = sp.head_block(sh, W, h)
    dh = sh.dh
    assert B.shape == (4 * dh, sh.d)
    assert np.array_equal(B[:dh], W["q"][2 * dh:3 * dh])
    assert np.array_equal(B[dh:2 * dh].T, W["o"][:, 2 * dh:3 * dh])
    assert np.array_equal(B[2 * dh:3 * dh], W["k"][dh:2 * dh])
    assert np.array_equal(B[3 * dh:], W["v"][dh:2 * dh])
    C = sp.channel_block(sh, W, 2)
    assert C.shape == (48, sh.d)
    assert np.array_equal(C[:16], W["gate"][32:48]) and np.array_equal(C[16:32], W["up"][32:48])
    assert np.array_equal(C[32:].T, W["down"][:, 32:48])
    # one candidate per query head and per channel group (Table 1)
    feats = sp.layer_features(sh, 0)
    assert len(feats) == sh.Hq + sh.n_chan_units
    assert [f.is_attention for f in feats] == [True] * sh.Hq + [False] * sh.n_chan_units


def test_gaussian_blocks_stay_inside_the_marchenko_pastur_edges():
    # i.i.d. N(0, 0.02^2) synthetic weights: the eigenvalues of a [n, d] block, scaled by
    # 1/d, fill [s^2 (1 - sqrt(n/d))^2, s^2 (1 + sqrt(n/d))^2] up to finite-size fluctuations
    sh = synth.tiny_shape(L=1, d=1024, Hq=4, Hkv=2, dh=32, df=256, chan_unit=32)
    W = sp.dense_f32(sh, 0)
    for B in (sp.head_block(sh, W, 1), sp.channel_block(sh, W, 3)):
        n = B.shape[0]
        lam = sp.eigenvalues(B, sh.d)
        r = np.sqrt(n / sh.d)
        lo, hi = synth.WEIGHT_SIGMA ** 2 * (1 - r) ** 2, synth.WEIGHT_SIGMA ** 2 * (1 + r) ** 2
        assert lam.min() > 0.8 * lo and lam.max() < 1.15 * hi
        assert lam.max() > 0.85 * hi and lam.min() < 1.3 * lo


def test_designed_power_law_spectrum_is_recovered():
    # singular values s_i = i^(-beta) give eigenvalues lambda_i ~ i^(-2 beta), whose counting
    # function #{lambda > x} ~ x^(-1 / (2 beta)): a Pareto tail of exponent 1 / (2 beta)
    for beta in (0.5, 0.25):
        n = 400
        s = np.arange(1, n + 1, dtype=np.float64) ** (-beta)
        W = _with_singular_values(s, n, n + 40, seed=9)
        f = sp.features(W, n + 40, 0, 1, False)
        assert f.alpha == pytest.approx(1.0 / (2 * beta), rel=0.03)
        assert f.spectral_norm == pytest.approx(1.0, rel=1e-10)
