"""Spectral descriptors of candidate units (Sec. 3.1 "Candidate Units and Spectral Features";
Appendix "Exact candidate feature construction", Eq. candidate-features). Test
infrastructure only.

For a candidate's weight block W (n_r x n_c) with singular values s_1 >= ... >= s_n the
eigenvalues of its normalized Gram matrix are lambda_i = s_i^2 / d_in. Features:

* the Pareto tail exponent alpha^ = (mean_i log(lambda_i / lambda_min))^-1 over the
  eigenvalues lambda_i >= lambda_min (maximum likelihood, Clauset et al. 2009), with
  lambda_min the value that minimizes the Kolmogorov-Smirnov distance between the tail and
  the fitted law P(x) = 1 - (x / lambda_min)^-alpha^;
* SETOL = sum of the tail eigenvalues / sum of all eigenvalues;
* effective rank r_eff = exp(-sum_i p_i log p_i), p_i = lambda_i / sum_j lambda_j;
* the spectral norm ||W||_2 = s_1.

Candidate blocks: an attention head h stacks its own Q rows, the O columns it feeds
(transposed), and the K and V rows of its KV group g(h) = h // g; a channel group G stacks
its gate rows, up rows and down columns (transposed). All blocks are [rows, d].

Readings (the paper leaves them open): d_in = d, the width all stacked pieces share (only
the eigenvalues' scale depends on it; alpha^, SETOL and r_eff are scale-free); the
candidates for lambda_min are the distinct eigenvalues below the largest one (a tail of
at least two values), ties in the KS distance go to the smaller lambda_min; the weights
are the synthetic model's unquantized FP32 ones (the paper reads the BF16 checkpoint); the
salience feature S_h needs calibration prompts and is not computed here.

Pins (tests/test_oracle_spectral.py): r_eff closed forms (equal eigenvalues give n, one
nonzero eigenvalue gives 1); the spectral norm against numpy's matrix 2-norm and a matrix
built from known singular values; alpha^ against scipy's Pareto maximum-likelihood fit, and
near the true exponent on a stratified Pareto sample; the KS distance against
scipy.stats.kstest; lambda_min against a brute-force scan with kstest; SETOL hand cases;
scale invariance; candidate blocks against the projections they come from; the
Marchenko-Pastur edges of i.i.d. Gaussian blocks.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

import synth
from . import weights as wts


# --------------------------------------------------------------------------
# Candidate blocks (Appendix "Exact candidate feature construction")
# --------------------------------------------------------------------------

def dense_f32(shape, layer: int) -> dict:
    """The unquantized FP32 projections of a layer, PyTorch [out, in] layout."""
    out = {}
    for name in wts.PROJ_NAMES:
        tid, rows, cols = wts.proj_dims(shape, name)
        out[name] = synth.weight_f32(shape.seed, tid, layer, rows, cols)
    return out


def head_block(shape, W: dict, h: int) -> np.ndarray:
    """[W_Q,h ; W_O,h^T ; W_K,g(h) ; W_V,g(h)]: [4 d_h, d]."""
    dh, j = shape.dh, h // shape.g
    return np.concatenate([W["q"][h * dh:(h + 1) * dh], W["o"][:, h * dh:(h + 1) * dh].T,
                           W["k"][j * dh:(j + 1) * dh], W["v"][j * dh:(j + 1) * dh]], axis=0)


def channel_block(shape, W: dict, unit: int) -> np.ndarray:
    """[W_gate,G ; W_up,G ; W_down,G^T] for channel group G = unit: [3 chan_unit, d]."""
    c0, c1 = unit * shape.chan_unit, (unit + 1) * shape.chan_unit
    return np.concatenate([W["gate"][c0:c1], W["up"][c0:c1], W["down"][:, c0:c1].T], axis=0)


# --------------------------------------------------------------------------
# Spectral statistics (Sec. 3.1)
# --------------------------------------------------------------------------

def eigenvalues(block: np.ndarray, d_in: int) -> np.ndarray:
    """lambda_i = s_i^2 / d_in in descending order (float64)."""
    s = np.linalg.svd(np.asarray(block, dtype=np.float64), compute_uv=False)
    return s * s / float(d_in)


def effective_rank(lam: np.ndarray) -> float:
    lam = np.asarray(lam, dtype=np.float64)
    p = lam[lam > 0] / np.sum(lam)
    return float(np.exp(-np.sum(p * np.log(p))))


def tail_alpha(lam: np.ndarray, lam_min: float) -> float:
    """Maximum-likelihood Pareto exponent of the eigenvalues >= lam_min."""
    t = np.asarray(lam, dtype=np.float64)
    t = t[t >= lam_min]
    return float(len(t) / np.sum(np.log(t / lam_min)))


def ks_distance(lam: np.ndarray, lam_min: float, alpha: float) -> float:
    """sup_x |S(x) - P(x)| over the tail, S its empirical CDF, P(x) = 1 - (x / lam_min)^-alpha."""
    t = np.sort(np.asarray(lam, dtype=np.float64)[np.asarray(lam) >= lam_min])
    n = len(t)
    P = 1.0 - (t / lam_min) ** (-alpha)
    i = np.arange(1, n + 1, dtype=np.float64)
    return float(max(np.max(i / n - P), np.max(P - (i - 1) / n)))


def setol(lam: np.ndarray, lam_min: float) -> float:
    lam = np.asarray(lam, dtype=np.float64)
    return float(np.sum(lam[lam >= lam_min]) / np.sum(lam))


def fit_tail(lam: np.ndarray):
    """(lambda_min, alpha^, D): the KS-minimizing lower cutoff and its exponent."""
    lam = np.asarray(lam, dtype=np.float64)
    vals = np.unique(lam[lam > 0])
    best = None
    for x in vals[:-1]:  # keep at least two distinct values in the tail
        a = tail_alpha(lam, x)
        D = ks_distance(lam, x, a)
        if best is None or D < best[2]:
            best = (float(x), a, D)
    return best


@dataclass
class Features:
    alpha: float
    r_eff: float
    spectral_norm: float
    setol: float
    lam_min: float
    ks: float
    layer_pos: float  # layer index / (L - 1), 0 for one layer
    is_attention: bool


def features(block: np.ndarray, d_in: int, layer: int, L: int, is_attention: bool) -> Features:
    lam = eigenvalues(block, d_in)
    lam_min, a, D = fit_tail(lam)
    return Features(alpha=a, r_eff=effective_rank(lam), spectral_norm=float(np.sqrt(lam[0] * d_in)),
                    setol=setol(lam, lam_min), lam_min=lam_min, ks=D,
                    layer_pos=layer / (L - 1) if L > 1 else 0.0, is_attention=is_attention)


def layer_features(shape, layer: int) -> list:
    """Features of every candidate of a layer: the H_q heads, then the channel groups."""
    W = dense_f32(shape, layer)
    out = [features(head_block(shape, W, h), shape.d, layer, shape.L, True) for h in range(shape.Hq)]
    out += [features(channel_block(shape, W, u), shape.d, layer, shape.L, False)
            for u in range(shape.n_chan_units)]
    return out
