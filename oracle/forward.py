"""Plain FP32 Llama-style decoder forward with masks applied as zeros. Test infrastructure only.

What the path computes (the paper fixes the architecture family, Sec. 3.3 and
the Limitations: decoder-only Transformers with grouped-query attention and
SwiGLU feed-forward blocks; the Llama-3 shapes of Table 1). Per layer and token:

    x^   = RMSNorm(x) * gamma_attn
    q, k, v = W~q x^, W~k x^, W~v x^          then rotary embedding on q, k
    o_h  = softmax(q_h K_j^T / sqrt(d_h)) V_j   for query head h in group j = h // g
    x    = x + W~o [o_1; ...; o_Hq]
    x^   = RMSNorm(x) * gamma_mlp
    x    = x + W~down (SiLU(W~gate x^) * (W~up x^))

and after the last layer logits = W_lm RMSNorm(x) * gamma_final (LM head dense,
Sec. 3.3). Readings (the paper is silent): RMSNorm eps 1e-5; rotary embedding
in the rotate-half convention with base 500,000 and frequencies
base^(-2i/d_h); prior KV-cache entries are already rotated; decode inputs are
teacher-forced vectors (no token feedback); new K/V are kept in FP32 here.

The mask enters only through ``oracle.weights.dense_zeroed`` (mask-as-zero).
``compact=True`` runs the same equations on the packed panels of
``oracle.pack`` instead; the two must agree (zero rows contribute zero). A mask
may keep single query heads (``keep_qheads``): the dropped heads' Q rows and O
columns are zero, and the compacted step maps each kept head to the position
of its KV head among the kept groups. A shape with ``quant_group`` > 0 runs on
groupwise-quantized weights (one BF16 scale per row and group of columns).

Pins: softmax against scipy.special.softmax, rotary embedding against complex
multiplication and its relative-position property, a single-key attention
returning V exactly, identical keys giving uniform attention, an empty mask
leaving the residual unchanged, all-keep equal to the unmasked forward,
mask-as-zero equal to compacted execution, and causal prefill equal to
step-by-step decode; the same two equalities with ragged query-head masks and
on groupwise stores, and a planted wrong query-to-KV map failing them.
"""
from __future__ import annotations

import numpy as np

import synth
from . import weights as wts
from .pack import kept_qheads, pack_layer
from .quant import dequantize


def rmsnorm(x, gamma, eps):
    x = np.asarray(x)
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return (x / np.sqrt(ms + x.dtype.type(eps))) * gamma


def silu(a):
    with np.errstate(over="ignore"):
        return a / (a.dtype.type(1) + np.exp(-a))


def rope_cos_sin(positions, dh, theta):
    """cos, sin [P, d_h/2] in float64 for angles pos * theta^(-2i/d_h)."""
    i = np.arange(dh // 2, dtype=np.float64)
    inv_freq = np.power(np.float64(theta), -2.0 * i / dh)
    ang = np.asarray(positions, dtype=np.float64)[:, None] * inv_freq[None, :]
    return np.cos(ang), np.sin(ang)


def apply_rope(v, cos, sin):
    """Rotate-half rotary embedding of v [..., d_h] with cos/sin broadcastable to [..., d_h/2]."""
    h = v.shape[-1] // 2
    a, b = v[..., :h], v[..., h:]
    c, s = cos.astype(v.dtype), sin.astype(v.dtype)
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def softmax(s, axis=-1):
    m = np.max(s, axis=axis, keepdims=True)
    e = np.exp(s - m)
    return e / np.sum(e, axis=axis, keepdims=True)


def attend(q, K, V, g, gmap=None):
    """q [Hq, d_h], K/V [Hkv, T, d_h] -> o [Hq, d_h] (GQA: head h reads group h // g, or
    the KV row ``gmap[h]`` when given)."""
    Hq, dh = q.shape
    o = np.empty_like(q)
    scale = q.dtype.type(1.0 / np.sqrt(dh))
    for h in range(Hq):
        j = h // g if gmap is None else gmap[h]
        p = softmax((K[j] @ q[h]) * scale)
        o[h] = p @ V[j]
    return o


def layer_step(shape, W, x, Kc, Vc, pos):
    """One decode step of one layer on dense (zeroed) weights.

    x [d]; Kc/Vc [H_kv, T, d_h] cache of earlier positions; returns (x_out, k [H_kv,d_h], v).
    """
    dt = x.dtype
    Hq, Hkv, dh = shape.Hq, shape.Hkv, shape.dh
    xn = rmsnorm(x, W["g_attn"], shape.eps)
    q = (W["q"] @ xn).reshape(Hq, dh)
    k = (W["k"] @ xn).reshape(Hkv, dh)
    v = (W["v"] @ xn).reshape(Hkv, dh)
    c, s = rope_cos_sin([pos], dh, shape.rope_theta)
    q, k = apply_rope(q, c, s), apply_rope(k, c, s)
    K = np.concatenate([Kc, k[:, None, :]], axis=1)
    V = np.concatenate([Vc, v[:, None, :]], axis=1)
    o = attend(q, K, V, shape.g).reshape(-1)
    x1 = x + W["o"] @ o
    xn2 = rmsnorm(x1, W["g_mlp"], shape.eps)
    h = silu(W["gate"] @ xn2) * (W["up"] @ xn2)
    x2 = x1 + W["down"] @ h
    return x2.astype(dt), k, v


def compact_weights(shape, lq, keep_groups, keep_chans, dtype=np.float32, keep_qheads=None):
    """Dequantized packed panels plus the row roles of the qkv panel: per kept group its
    kept query heads' row blocks, then K, then V (``oracle.pack``); ``gmap`` gives each
    kept query head the position of its KV head among the kept groups."""
    P = pack_layer(shape, lq, keep_groups, keep_chans, keep_qheads)
    qh = set(kept_qheads(shape, keep_groups, keep_qheads))
    blocks, q_blk, k_blk, v_blk, gmap = 0, [], [], [], []
    for i, j in enumerate(keep_groups):
        for h in range(j * shape.g, (j + 1) * shape.g):
            if h in qh:
                q_blk.append(blocks)
                gmap.append(i)
                blocks += 1
        k_blk.append(blocks)
        v_blk.append(blocks + 1)
        blocks += 2
    return dict(qkv=dequantize(P["qkv_w"], P["qkv_s"], dtype),
                o=dequantize(P["o_w"], P["o_s"], dtype),
                gu=dequantize(P["gu_w"], P["gu_s"], dtype),
                down=dequantize(P["down_w"], P["down_s"], dtype),
                g_attn=lq.g_attn.astype(dtype), g_mlp=lq.g_mlp.astype(dtype),
                m_kv=len(keep_groups), q_blk=q_blk, k_blk=k_blk, v_blk=v_blk, gmap=gmap)


def layer_step_compact(shape, P, x, Kc, Vc, pos):
    """The same step on packed panels; Kc/Vc hold only the kept groups [m_kv, T, d_h]."""
    dt = x.dtype
    g, dh, m = shape.g, shape.dh, P["m_kv"]
    xn = rmsnorm(x, P["g_attn"], shape.eps)
    y = (P["qkv"] @ xn).reshape(-1, dh)
    c, s = rope_cos_sin([pos], dh, shape.rope_theta)
    q = apply_rope(y[P["q_blk"]], c, s)
    k = apply_rope(y[P["k_blk"]], c, s)
    v = y[P["v_blk"]]
    K = np.concatenate([Kc, k[:, None, :]], axis=1)
    V = np.concatenate([Vc, v[:, None, :]], axis=1)
    o = attend(q, K, V, g, P["gmap"]).reshape(-1) if len(P["gmap"]) else np.zeros(0, dt)
    x1 = x + P["o"] @ o
    xn2 = rmsnorm(x1, P["g_mlp"], shape.eps)
    z = P["gu"] @ xn2
    h = silu(z[0::2]) * z[1::2]
    x2 = x1 + P["down"] @ h
    return x2.astype(dt), k, v


def prior_cache(shape, layer, kv_seed, t_prior, groups=None, dtype=np.float32):
    """Synthetic prior K/V (BF16 N(0,1) widened) [len(groups), t_prior, d_h]."""
    groups = range(shape.Hkv) if groups is None else groups
    K = np.stack([synth.bf16_to_f32(synth.kv_prior_bf16(kv_seed, layer, j, t_prior, shape.dh, synth.T_KCACHE))
                  for j in groups]) if len(groups) else np.zeros((0, t_prior, shape.dh), np.float32)
    V = np.stack([synth.bf16_to_f32(synth.kv_prior_bf16(kv_seed, layer, j, t_prior, shape.dh, synth.T_VCACHE))
                  for j in groups]) if len(groups) else np.zeros((0, t_prior, shape.dh), np.float32)
    return K.astype(dtype), V.astype(dtype)


def decode(shape, mask, x_steps, t_prior, kv_seed, compact=False, dtype=np.float32,
           layers=None, x_in=None, prior=None):
    """Teacher-forced batch-1 decode of len(x_steps) steps.

    x_steps [S, d] float inputs (the BF16 step vectors widened). Processes the
    model layer by layer (each step's layer input is that step's previous layer
    output, so the loop order does not change the result). Returns the residual
    stream after the last processed layer [S, d].
    ``layers`` restricts to a sub-range; ``x_in`` then supplies its input.
    ``prior`` (optional) maps a layer to its dense cache (K, V) [H_kv, t_prior, d_h] (for
    decoding after a prefill) instead of the synthetic prior tokens.
    """
    X = np.array(x_steps if x_in is None else x_in, dtype=dtype)
    S = X.shape[0]
    for layer in (range(shape.L) if layers is None else layers):
        lq = wts.gen_layer(shape, layer)
        kg, kc, qh = mask.keep_groups[layer], mask.keep_chans[layer], mask.qheads(shape, layer)
        if prior is not None:
            Kd, Vd = prior(layer)
            Kd, Vd = np.asarray(Kd, dtype), np.asarray(Vd, dtype)
        if compact:
            W = compact_weights(shape, lq, kg, kc, dtype, qh)
            Kc, Vc = (Kd[kg], Vd[kg]) if prior is not None else prior_cache(shape, layer, kv_seed, t_prior, kg, dtype)
        else:
            W = wts.dense_zeroed(shape, lq, kg, kc, dtype, qh)
            Kc, Vc = (Kd, Vd) if prior is not None else prior_cache(shape, layer, kv_seed, t_prior, None, dtype)
        nkv = Kc.shape[0]
        Kall = np.zeros((nkv, t_prior + S, shape.dh), dtype)
        Vall = np.zeros_like(Kall)
        Kall[:, :t_prior], Vall[:, :t_prior] = Kc, Vc
        for t in range(S):
            T = t_prior + t
            f = layer_step_compact if compact else layer_step
            X[t], k, v = f(shape, W, X[t], Kall[:, :T], Vall[:, :T], T)
            Kall[:, T], Vall[:, T] = k, v
        del W
    return X


def decode_sessions(shape, mask, x_steps, t_priors, kv_seeds, dtype=np.float32):
    """Teacher-forced decode of several independent sessions on one mask (Sec. 3.3: the
    turns that share a mask share its plan; each keeps its own KV cache and position).

    x_steps [S, n, d]; session i starts from its synthetic prior cache of t_priors[i]
    tokens keyed by kv_seeds[i]. Each session is exactly ``decode`` of its own inputs;
    the loop visits layers outermost only so that a layer's weights are made once.
    Returns [S, n, d].
    """
    X = np.array(x_steps, dtype=dtype)
    S, n = X.shape[0], X.shape[1]
    for layer in range(shape.L):
        lq = wts.gen_layer(shape, layer)
        W = wts.dense_zeroed(shape, lq, mask.keep_groups[layer], mask.keep_chans[layer], dtype,
                             mask.qheads(shape, layer))
        for i in range(n):
            tp = int(t_priors[i])
            Kc, Vc = prior_cache(shape, layer, kv_seeds[i], tp, None, dtype)
            Kall = np.zeros((Kc.shape[0], tp + S, shape.dh), dtype)
            Vall = np.zeros_like(Kall)
            Kall[:, :tp], Vall[:, :tp] = Kc, Vc
            for t in range(S):
                T = tp + t
                X[t, i], k, v = layer_step(shape, W, X[t, i], Kall[:, :T], Vall[:, :T], T)
                Kall[:, T], Vall[:, T] = k, v
        del W
    return X


def final_logits(shape, x, dtype=np.float32, rows=None, chunk=8192):
    """logits = W_lm RMSNorm(x) gamma_final for x [S, d]; ``rows`` selects vocabulary rows."""
    xn = rmsnorm(np.asarray(x, dtype=dtype), wts.gamma_final(shape).astype(dtype), shape.eps)
    if rows is not None:
        out = np.empty((xn.shape[0], len(rows)), dtype)
        for i, r in enumerate(rows):
            out[:, i] = xn @ wts.lm_head_f32(shape, int(r), 1)[0].astype(dtype)
        return out
    out = np.empty((xn.shape[0], shape.vocab), dtype)
    for r0 in range(0, shape.vocab, chunk):
        n = min(chunk, shape.vocab - r0)
        out[:, r0:r0 + n] = xn @ wts.lm_head_f32(shape, r0, n).astype(dtype).T
    return out


# --------------------------------------------------------------------------
# Prefill: causal attention over a whole prompt (positions 0 .. T-1).
# --------------------------------------------------------------------------

def layer_prefill(shape, W, X):
    """X [T, d] -> (X_out [T, d], K [H_kv, T, d_h], V) on dense (zeroed) weights."""
    T = X.shape[0]
    Hq, Hkv, dh, g = shape.Hq, shape.Hkv, shape.dh, shape.g
    Xn = rmsnorm(X, W["g_attn"], shape.eps)
    Q = (Xn @ W["q"].T).reshape(T, Hq, dh)
    K = (Xn @ W["k"].T).reshape(T, Hkv, dh)
    V = (Xn @ W["v"].T).reshape(T, Hkv, dh)
    c, s = rope_cos_sin(np.arange(T), dh, shape.rope_theta)
    Q = apply_rope(Q, c[:, None, :], s[:, None, :])
    K = apply_rope(K, c[:, None, :], s[:, None, :])
    causal = np.triu(np.ones((T, T), dtype=bool), 1)
    O = np.empty_like(Q)
    scale = X.dtype.type(1.0 / np.sqrt(dh))
    for h in range(Hq):
        j = h // g
        S = (Q[:, h, :] @ K[:, j, :].T) * scale
        S[causal] = -np.inf
        O[:, h, :] = softmax(S, axis=-1) @ V[:, j, :]
    X1 = X + O.reshape(T, Hq * dh) @ W["o"].T
    Xn2 = rmsnorm(X1, W["g_mlp"], shape.eps)
    H = silu(Xn2 @ W["gate"].T) * (Xn2 @ W["up"].T)
    X2 = X1 + H @ W["down"].T
    return X2.astype(X.dtype), K.transpose(1, 0, 2).copy(), V.transpose(1, 0, 2).copy()


def prefill(shape, mask, X, dtype=np.float32, layers=None):
    """Causal prefill of a prompt X [T, d]; returns (residual [T, d], per-layer (K, V))."""
    X = np.array(X, dtype=dtype)
    kv = []
    for layer in (range(shape.L) if layers is None else layers):
        lq = wts.gen_layer(shape, layer)
        W = wts.dense_zeroed(shape, lq, mask.keep_groups[layer], mask.keep_chans[layer], dtype,
                             mask.qheads(shape, layer))
        X, K, V = layer_prefill(shape, W, X)
        kv.append((K, V))
    return X, kv
