"""Pins of the oracle's forward pass (mask-as-zero decoder)."""
import numpy as np
import pytest
import scipy.special
import torch

import synth
from oracle import forward as fw
from oracle import maskc, weights


def test_softmax_matches_scipy():
    s = np.random.default_rng(0).standard_normal((7, 33)) * 10
    assert np.allclose(fw.softmax(s), scipy.special.softmax(s, axis=-1), rtol=1e-12, atol=0)


def test_silu_matches_expit():
    a = np.linspace(-30, 30, 1001)
    assert np.allclose(fw.silu(a), a * scipy.special.expit(a), rtol=1e-12, atol=1e-300)


def test_rope_is_complex_rotation():
    rng = np.random.default_rng(1)
    dh, theta = 16, 500000.0
    v = rng.standard_normal((3, dh))
    pos = np.array([0, 5, 4099])
    c, s = fw.rope_cos_sin(pos, dh, theta)
    got = fw.apply_rope(v, c, s)
    z = v[:, : dh // 2] + 1j * v[:, dh // 2:]
    ang = pos[:, None] * theta ** (-2.0 * np.arange(dh // 2) / dh)[None, :]
    w = z * np.exp(1j * ang)
    assert np.allclose(got, np.concatenate([w.real, w.imag], axis=-1), atol=1e-12)
    # position 0 is the identity; frequency 0 turns by exactly the position
    assert np.allclose(got[0], v[0])
    assert np.isclose(c[2, 0], np.cos(4099.0)) and np.isclose(s[2, 0], np.sin(4099.0))


def test_rope_relative_position():
    rng = np.random.default_rng(2)
    dh = 32
    q, k = rng.standard_normal(dh), rng.standard_normal(dh)

    def dot(m, n):
        cm, sm = fw.rope_cos_sin([m], dh, 500000.0)
        cn, sn = fw.rope_cos_sin([n], dh, 500000.0)
        return fw.apply_rope(q[None], cm, sm)[0] @ fw.apply_rope(k[None], cn, sn)[0]

    assert np.isclose(dot(10, 3), dot(110, 103), rtol=1e-9)
    assert not np.isclose(dot(10, 3), dot(10, 4), rtol=1e-3)


def test_attend_matches_torch_sdpa_gqa():
    rng = np.random.default_rng(3)
    Hq, Hkv, T, dh = 8, 2, 37, 16
    q = rng.standard_normal((Hq, dh))
    K = rng.standard_normal((Hkv, T, dh))
    V = rng.standard_normal((Hkv, T, dh))
    got = fw.attend(q, K, V, Hq // Hkv)
    g = Hq // Hkv
    Kt = torch.from_numpy(K).repeat_interleave(g, dim=0)  # query head h reads KV head h // g
    Vt = torch.from_numpy(V).repeat_interleave(g, dim=0)
    want = torch.nn.functional.scaled_dot_product_attention(torch.from_numpy(q)[:, None, :], Kt, Vt)[:, 0, :]
    assert np.allclose(got, want.numpy(), atol=1e-12)


def test_attend_single_key_and_identical_keys():
    rng = np.random.default_rng(4)
    q = rng.standard_normal((4, 8)) * 5
    K = rng.standard_normal((2, 1, 8))
    V = rng.standard_normal((2, 1, 8))
    o = fw.attend(q, K, V, 2)
    assert np.array_equal(o[0], V[0, 0]) and np.array_equal(o[3], V[1, 0])
    K2 = np.repeat(K, 5, axis=1)
    V2 = rng.standard_normal((2, 5, 8))
    o2 = fw.attend(q, K2, V2, 2)
    assert np.allclose(o2[1], V2[0].mean(axis=0), atol=1e-12)


def test_rmsnorm_scale_invariance_and_eps():
    rng = np.random.default_rng(5)
    x = rng.standard_normal(64)
    g = 1 + 0.1 * rng.standard_normal(64)
    y = fw.rmsnorm(x, g, 1e-5)
    # eps sits inside the root: scaling x by c is the same as dividing eps by c^2
    assert np.allclose(fw.rmsnorm(37.0 * x, g, 1e-5), fw.rmsnorm(x, g, 1e-5 / 37.0 ** 2), rtol=1e-12)
    assert np.allclose(fw.rmsnorm(37.0 * x, g, 1e-5), y, rtol=1e-5)
    assert np.isclose(np.sqrt(np.mean((y / g) ** 2)), 1.0, rtol=1e-5)
    tiny = 1e-9 * x  # mean square far below eps: output ~ x / sqrt(eps)
    assert np.allclose(fw.rmsnorm(tiny, g, 1e-5), tiny / np.sqrt(1e-5) * g, rtol=1e-6)


def _setup(shape, seed=3):
    sc = synth.mask_scores_u32(seed, shape.L, shape.n_units)
    return maskc.compile_mask(shape, sc, synth.layer_target_u24(seed, shape.L))


def _steps(shape, S, seed=11):
    return synth.bf16_to_f32(synth.step_inputs_bf16(seed, S, 1, shape.d))[:, 0]


def test_empty_mask_is_identity_layer():
    sh = synth.tiny_shape(L=1)
    m = maskc.explicit(sh, [[]], [[]])
    x = _steps(sh, 3)
    X = fw.decode(sh, m, x, 4, 7, dtype=np.float64)
    assert np.array_equal(X, x.astype(np.float64))


def test_all_keep_equals_unmasked_dense():
    sh = synth.tiny_shape(L=1)
    lq = weights.gen_layer(sh, 0)
    m = maskc.all_keep(sh)
    W = weights.dense_zeroed(sh, lq, m.keep_groups[0], m.keep_chans[0], np.float64)
    for name in weights.PROJ_NAMES:
        from oracle.quant import dequantize_rows
        assert np.array_equal(W[name], dequantize_rows(lq.q[name], lq.s[name], np.float64))


@pytest.mark.parametrize("dtype,tol", [(np.float64, 1e-12), (np.float32, 2e-5)])
def test_mask_as_zero_equals_compacted(dtype, tol):
    sh = synth.tiny_shape(L=3)
    m = _setup(sh)
    x = _steps(sh, 5)
    Xz = fw.decode(sh, m, x, 9, 7, dtype=dtype)
    Xc = fw.decode(sh, m, x, 9, 7, compact=True, dtype=dtype)
    assert np.linalg.norm(Xz - Xc) <= tol * np.linalg.norm(Xz)
    # and the mask matters at all
    Xd = fw.decode(sh, maskc.all_keep(sh), x, 9, 7, dtype=dtype)
    assert np.linalg.norm(Xd - Xz) > 1e-3 * np.linalg.norm(Xz)


def test_layer1_mask_as_zero_equals_compacted():
    sh = synth.LAYER1
    m = _setup(sh, 1000)
    x = _steps(sh, 4)
    Xz = fw.decode(sh, m, x, 128, 7, dtype=np.float64)
    Xc = fw.decode(sh, m, x, 128, 7, compact=True, dtype=np.float64)
    assert np.abs(Xz - Xc).max() <= 1e-12 * np.abs(Xz).max()


def test_prefill_equals_stepwise_decode():
    sh = synth.tiny_shape(L=2)
    m = _setup(sh)
    T = 6
    X = _steps(sh, T).astype(np.float64)
    Xp, kv = fw.prefill(sh, m, X, dtype=np.float64)
    Xd = fw.decode(sh, m, X, 0, 7, dtype=np.float64)  # empty prior cache
    assert np.allclose(Xp, Xd, rtol=1e-10, atol=1e-10)


def test_prefill_attention_matches_torch_causal_and_is_causal():
    sh = synth.tiny_shape(L=1)
    m = maskc.all_keep(sh)
    T = 9
    X = _steps(sh, T).astype(np.float64)
    Xp, _ = fw.prefill(sh, m, X, dtype=np.float64)
    X2 = X.copy()
    X2[-1] += 1.0
    Xp2, _ = fw.prefill(sh, m, X2, dtype=np.float64)
    assert np.array_equal(Xp[:-1], Xp2[:-1]) and not np.allclose(Xp[-1], Xp2[-1])
    # the attention core against torch's causal SDPA
    rng = np.random.default_rng(6)
    Q = rng.standard_normal((4, T, 8))
    K = rng.standard_normal((2, T, 8))
    V = rng.standard_normal((2, T, 8))
    causal = np.triu(np.ones((T, T), dtype=bool), 1)
    out = np.empty_like(Q)
    for h in range(4):
        S = Q[h] @ K[h // 2].T / np.sqrt(8)
        S[causal] = -np.inf
        out[h] = fw.softmax(S) @ V[h // 2]
    want = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(Q), torch.from_numpy(K).repeat_interleave(2, 0), torch.from_numpy(V).repeat_interleave(2, 0),
        is_causal=True)
    assert np.allclose(out, want.numpy(), atol=1e-12)


def test_decode_first_step_single_prior_free_layer_reduces_to_v():
    # H_kv = 1, no prior: the one key is the token itself, softmax(1) = 1 and o = v
    sh = synth.tiny_shape(L=1, Hq=2, Hkv=1, d=64, dh=16, df=32, chan_unit=8)
    lq = weights.gen_layer(sh, 0)
    m = maskc.all_keep(sh)
    W = weights.dense_zeroed(sh, lq, m.keep_groups[0], m.keep_chans[0], np.float64)
    x = _steps(sh, 1)[0].astype(np.float64)
    xn = fw.rmsnorm(x, W["g_attn"], sh.eps)
    v = W["v"] @ xn
    Wz = dict(W)
    Wz["gate"] = np.zeros_like(W["gate"])  # silence the MLP: the layer adds W_o [v; v]
    x1, _, _ = fw.layer_step(sh, Wz, x, np.zeros((1, 0, 16)), np.zeros((1, 0, 16)), 0)
    assert np.allclose(x1, x + W["o"] @ np.concatenate([v, v]), rtol=1e-12, atol=1e-12)


def test_planted_gqa_mistake_is_caught():
    # a wrong query-head to group map (h % H_kv instead of h // g) must fail the SDPA pin
    rng = np.random.default_rng(7)
    q = rng.standard_normal((8, 16))
    K = rng.standard_normal((2, 11, 16))
    V = rng.standard_normal((2, 11, 16))
    right = fw.attend(q, K, V, 4)
    wrong = np.stack([fw.softmax(K[h % 2] @ q[h] / 4.0) @ V[h % 2] for h in range(8)])
    assert not np.allclose(right, wrong)


def test_decode_sessions_is_per_session_decode():
    # sessions sharing a mask are independent: each equals its own batch-1 decode (same
    # arithmetic, so bit-identical), and sessions with different caches differ
    sh = synth.tiny_shape(L=2)
    m = _setup(sh)
    x = np.stack([_steps(sh, 3) * (1 + i) for i in range(3)], axis=1)  # [S, n, d]
    tps, seeds = [5, 9, 1], [7, 8, 7]
    X = fw.decode_sessions(sh, m, x, tps, seeds, dtype=np.float64)
    for i in range(3):
        Xi = fw.decode(sh, m, x[:, i], tps[i], seeds[i], dtype=np.float64)
        assert np.array_equal(X[:, i], Xi)
    Y = fw.decode_sessions(sh, m, np.repeat(x[:, :1], 2, axis=1), [5, 5], [7, 8], dtype=np.float64)
    assert not np.allclose(Y[:, 0], Y[:, 1])
