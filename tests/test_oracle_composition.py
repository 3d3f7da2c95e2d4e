"""Hand-worked pins of how the oracle composes one decoder layer and the final norm + LM head.

The per-piece pins (softmax, SiLU, rotary, GQA attention, RMSNorm) cannot see how the
pieces are wired together: which projection gets the SiLU, which gain each RMSNorm
uses, which residual the MLP adds to. Here one layer with hand-picked weights is worked
out on paper (eps = 0 so every intermediate is exact), and the oracle must reproduce
it. Each plausible wiring mistake is planted in a copy of the layer step and must miss
the hand result. The layer follows Sec. 3.3 (a Llama-style GQA + SwiGLU decoder) and
Appendix Eq. flop-mlp (gate row, up row and down column of a channel act together).
"""
import math

import numpy as np
import pytest

import synth
from oracle import forward as fw
from oracle import weights

# d = 4, one KV head with g = 2 query heads of d_h = 2, two SwiGLU channels, eps = 0
SH = synth.ModelShape(L=1, d=4, Hq=2, Hkv=1, dh=2, df=2, vocab=0, chan_unit=1, eps=0.0)


def _silu(a):
    return a / (1.0 + math.exp(-a))


def _hand_weights(q_zero=False):
    W = {
        "g_attn": np.array([1.0, 2.0, 3.0, 4.0]),
        "g_mlp": np.array([2.0, 1.0, 1.0, 1.0]),
        # q: identity rows (or zero for the uniform-attention case), k reads x^ columns 2, 3
        "q": np.zeros((4, 4)) if q_zero else np.eye(4),
        "k": np.array([[0.0, 0, 1, 0], [0, 0, 0, 1]]),
        "v": np.array([[1.0, 0, 0, 0], [0, 1, 0, 0]]),
        "o": np.array([[-1.0, -1, -1, 0], [0, 0, 0, 0], [0, 0, 0, 0], [0, 0, 0, 0]]),
        "gate": np.array([[1.0, 0, 0, 0], [0, 0, 1, 1]]),
        "up": np.array([[0.0, 1, 0, 0], [0, 0, 0, -0.5]]),
        "down": np.array([[1.0, 0], [0, 1], [0, 0], [0, 0]]),
    }
    return W


# Worked by hand. x = (2, 2, 2, 2): rms 2, x / rms = (1, 1, 1, 1), x^ = gamma_attn = (1, 2, 3, 4).
# v = (1, 2). Case A (position 0, empty cache): the only key is the token's own, so each
# head's output is v and o = (1, 2, 1, 2). Case B (position 1, one prior key, q = 0): both
# keys score 0, the weights are 1/2 each, o_h = (v + v_prior) / 2 with v_prior = (3, -2),
# i.e. (2, 0) for both heads. Either way W_o o = (-4, 0, 0, 0) and x1 = (-2, 2, 2, 2).
# x1: rms 2, x1 / rms = (-1, 1, 1, 1), x^2 = (-1, 1, 1, 1) * gamma_mlp = (-2, 1, 1, 1).
# gate x^2 = (-2, 2), up x^2 = (1, -0.5), h = (SiLU(-2) * 1, SiLU(2) * -0.5).
# x2 = x1 + W_down h = (-2 + SiLU(-2), 2 - 0.5 SiLU(2), 2, 2).
X = np.array([2.0, 2.0, 2.0, 2.0])
V_PRIOR = np.array([3.0, -2.0])
K_PRIOR = np.array([0.5, -7.0])
X2_HAND = np.array([-2.0 + _silu(-2.0), 2.0 - 0.5 * _silu(2.0), 2.0, 2.0])
K_NEW_HAND = np.array([3.0, 4.0])  # k = x^ columns 2, 3; rotary at position 0 is the identity
V_NEW_HAND = np.array([1.0, 2.0])


def _case(name):
    if name == "A":
        return _hand_weights(), np.zeros((1, 0, 2)), np.zeros((1, 0, 2)), 0
    return _hand_weights(q_zero=True), K_PRIOR.reshape(1, 1, 2), V_PRIOR.reshape(1, 1, 2), 1


@pytest.mark.parametrize("case", ["A", "B"])
def test_layer_step_matches_hand_worked_layer(case):
    W, Kc, Vc, pos = _case(case)
    x2, k, v = fw.layer_step(SH, W, X.copy(), Kc, Vc, pos)
    assert np.allclose(x2, X2_HAND, rtol=0, atol=1e-14)
    assert np.allclose(v[0], V_NEW_HAND, rtol=0, atol=1e-14)  # the value row is not rotated
    if pos == 0:
        assert np.allclose(k[0], K_NEW_HAND, rtol=0, atol=1e-14)


def test_prefill_of_one_token_matches_hand_worked_layer():
    W, _, _, _ = _case("A")
    X2, K, V = fw.layer_prefill(SH, W, X[None, :].copy())
    assert np.allclose(X2[0], X2_HAND, rtol=0, atol=1e-14)
    assert np.allclose(K[0, 0], K_NEW_HAND, atol=1e-14) and np.allclose(V[0, 0], V_NEW_HAND, atol=1e-14)


# ---- planted wiring mistakes: each copy differs from the oracle's step in one place
def _mutant(W, x, Kc, Vc, pos, mistake):
    xn = fw.rmsnorm(x, W["g_attn"], SH.eps)
    q = (W["q"] @ xn).reshape(SH.Hq, SH.dh)
    k = (W["k"] @ xn).reshape(SH.Hkv, SH.dh)
    v = (W["v"] @ xn).reshape(SH.Hkv, SH.dh)
    c, s = fw.rope_cos_sin([pos], SH.dh, SH.rope_theta)
    q, k = fw.apply_rope(q, c, s), fw.apply_rope(k, c, s)
    if mistake == "rope_on_v":
        v = fw.apply_rope(v, c, s)
    K = np.concatenate([Kc, k[:, None, :]], axis=1)
    V = np.concatenate([Vc, v[:, None, :]], axis=1)
    o = fw.attend(q, K, V, SH.g).reshape(-1)
    x1 = x + W["o"] @ o
    g2 = W["g_attn"] if mistake == "attn_gain_for_mlp" else W["g_mlp"]
    xn2 = x1 if mistake == "no_mlp_norm" else fw.rmsnorm(x1, g2, SH.eps)
    a, b = W["gate"] @ xn2, W["up"] @ xn2
    h = fw.silu(b) * a if mistake == "silu_on_up" else fw.silu(a) * b
    base = x if mistake == "mlp_residual_on_x" else x1
    return base + W["down"] @ h


@pytest.mark.parametrize("mistake", ["silu_on_up", "attn_gain_for_mlp", "mlp_residual_on_x", "no_mlp_norm",
                                     "rope_on_v"])
def test_planted_wiring_mistakes_miss_the_hand_result(mistake):
    case = "B" if mistake == "rope_on_v" else "A"  # the rotation is the identity at position 0
    W, Kc, Vc, pos = _case(case)
    assert np.allclose(_mutant(W, X.copy(), Kc, Vc, pos, "none"), X2_HAND, atol=1e-14)  # the copy is faithful
    assert not np.allclose(_mutant(W, X.copy(), Kc, Vc, pos, mistake), X2_HAND, atol=1e-3)


# ---- final norm + LM head
def test_final_logits_one_hot_picks_a_scaled_head_column():
    # x = c e_k with c^2 / d far above eps: RMSNorm(x) = sqrt(d) e_k (relative error ~ eps d / c^2),
    # so logits = sqrt(d) gamma_final[k] W_lm[:, k] (Sec. 3.3: the LM head stays dense)
    sh = synth.tiny_shape(L=1)
    gf = weights.gamma_final(sh).astype(np.float64)
    k = int(np.argmax(np.abs(gf - 1.0)))  # the gain furthest from 1, so a dropped gain shows
    assert abs(gf[k] - 1.0) > 0.02
    x = np.zeros((1, sh.d))
    x[0, k] = 1000.0
    got = fw.final_logits(sh, x, dtype=np.float64)[0]
    col = weights.lm_head_f32(sh, 0, sh.vocab)[:, k].astype(np.float64)
    want = math.sqrt(sh.d) * gf[k] * col
    assert np.allclose(got, want, rtol=1e-8, atol=0)
    # planted: no final gain, or the last layer's MLP gain in its place
    assert not np.allclose(got, math.sqrt(sh.d) * col, rtol=1e-3, atol=0)
    g_mlp = weights.gen_layer(sh, sh.L - 1).g_mlp.astype(np.float64)
    assert not np.allclose(got, math.sqrt(sh.d) * g_mlp[k] * col, rtol=1e-3, atol=0)
    # the sampled-rows path equals the full head
    rows = [0, 7, sh.vocab - 1]
    assert np.allclose(fw.final_logits(sh, x, dtype=np.float64, rows=rows)[0], got[rows], rtol=1e-12)
