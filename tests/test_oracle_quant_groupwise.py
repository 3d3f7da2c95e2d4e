"""Pins of the oracle's groupwise INT8 quantizer (the paper's group size 128 with BF16
scales, Table 1 and Appendix "Backing-store semantics"), the first step of the groupwise
variant of the path. CPU only."""
import numpy as np
import pytest

import synth
from oracle import quant


def test_bf16_rounding_ties_and_torch():
    torch = pytest.importorskip("torch")
    # exact ties go to the even 16-bit pattern
    u = np.array([0x3F808000, 0x3F818000, 0x3F80FFFF, 0x3F807FFF, 0xBF808000], np.uint32)
    got = quant.to_bf16(u.view(np.float32)).view(np.uint32)
    assert got.tolist() == [0x3F800000, 0x3F820000, 0x3F810000, 0x3F800000, 0xBF800000]
    x = np.random.default_rng(5).standard_normal(100000).astype(np.float32) * np.float32(1e-3)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(quant.to_bf16(x).view(np.uint32), ref.view(np.uint32))


def test_groupwise_hand_cases():
    s = np.float32(2.0 ** -10)  # exactly representable in BF16
    g0 = np.zeros(128, np.float32)
    g0[:6] = np.array([127, -127, 0.5, 1.5, -2.5, 3.25], np.float32) * s
    g1 = np.zeros(128, np.float32)  # a zero group in the same row
    q, sc = quant.quantize_groupwise(np.concatenate([g0, g1])[None, :])
    assert sc[0, 0] == s and sc[0, 1] == 0
    assert q[0, :6].tolist() == [127, -127, 0, 2, -2, 3]  # ties to even
    assert not q[0, 6:].any()


def _brute_nearest(w, s):
    """The integer k in [-127, 127] nearest to w / s (ties to even), by search."""
    k = np.arange(-127, 128, dtype=np.float64)
    out = np.empty(w.shape, np.int64)
    for i, (wi, si) in enumerate(zip(w.ravel(), s.ravel())):
        if si == 0:
            out.flat[i] = 0
            continue
        d = np.abs(wi / np.float64(si) - k)
        best = np.flatnonzero(d == d.min())
        out.flat[i] = int(k[best[0]]) if len(best) == 1 else int(k[best[np.argmin(np.abs(k[best]) % 2)]])
    return out


def test_groupwise_scales_and_codes_match_definition():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(11)
    w = (rng.standard_normal((6, 512)) * 0.02).astype(np.float32)
    w[2, 128:256] = 0  # a zero group
    q, s = quant.quantize_groupwise(w)
    a = np.abs(w.reshape(6, 4, 128)).max(axis=2)
    want = torch.from_numpy((a / np.float32(127)).astype(np.float32)).to(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(s.view(np.uint32), want.view(np.uint32))
    assert not (s.view(np.uint32) & 0xFFFF).any()  # every scale is a BF16 value
    sf = np.repeat(s, 128, axis=1)
    ref = _brute_nearest(w.astype(np.float64), sf)
    assert np.array_equal(q.astype(np.int64), ref)


def test_groupwise_error_bound_and_clamp():
    rng = np.random.default_rng(3)
    w = (rng.standard_normal((64, 1024)) * 0.02).astype(np.float32)
    q, s = quant.quantize_groupwise(w)
    sf = np.repeat(s, 128, axis=1)
    err = np.abs(quant.dequantize_groupwise(q, s) - w)
    clamped = np.abs(q) == 127
    inside = ~clamped | (np.abs(w) <= 127 * sf)
    assert (err[inside] <= 0.5 * sf[inside] * (1 + 2.0 ** -20) + 2.0 ** -24 * np.abs(w[inside])).all()
    # a BF16 scale rounded down can leave |w| / s just above 127: only then does the clamp act
    over = np.abs(w) > 127 * sf
    assert (np.abs(q[over]) == 127).all()
    assert (np.abs(w[over]) <= 127 * sf[over] * (1 + 2.0 ** -8)).all()


def test_groupwise_is_more_accurate_than_per_row_on_the_synthetic_weights():
    # 8B-shape gate rows of layer 0 (N(0, 0.02) from the counter-based generator): the
    # 128-column groups with BF16 scales reconstruct the weights, and a projection of an
    # RMS-normalized input, more closely than one FP32 scale per row
    sh = synth.LLAMA3_8B
    w = synth.weight_f32(sh.seed, synth.T_WGATE, 0, sh.df, sh.d, 0, 256)
    qr, sr = quant.quantize_rows(w)
    qg, sg = quant.quantize_groupwise(w)
    wr, wg = quant.dequantize_rows(qr, sr), quant.dequantize_groupwise(qg, sg)
    e_row = np.sqrt(np.mean((wr - w) ** 2))
    e_grp = np.sqrt(np.mean((wg - w) ** 2))
    assert e_grp < 0.8 * e_row
    x = np.random.default_rng(9).standard_normal(sh.d).astype(np.float64)
    y = w.astype(np.float64) @ x
    r_row = np.linalg.norm(wr.astype(np.float64) @ x - y) / np.linalg.norm(y)
    r_grp = np.linalg.norm(wg.astype(np.float64) @ x - y) / np.linalg.norm(y)
    assert r_grp < r_row


# ---------------------------------------------------------------------------
# Groupwise stores through the rest of the oracle: C regenerator, packing, forward.
# ---------------------------------------------------------------------------

def test_c_groupwise_quantizer_is_bit_identical():
    from oracle import cgen
    if not cgen.available():
        pytest.skip("no C compiler")
    rng = np.random.default_rng(3)
    w = (rng.standard_normal((40, 512)) * 0.02).astype(np.float32)
    w[5, 128:256] = 0  # a zero group
    w[7, :128] = np.float32(2.0 ** -10) * np.arange(-64, 64, dtype=np.float32) / np.float32(2)  # ties
    q, s = quant.quantize_groupwise(w)
    for r in range(w.shape[0]):
        qc, sc = cgen.quant_row_grouped(w[r], 128)
        assert np.array_equal(qc, q[r]) and np.array_equal(sc.view(np.uint32), s[r].view(np.uint32))
    # and the threaded regenerator against the numpy generator + quantizer
    sh = synth.LLAMA3_8B
    key = synth.stream_key(sh.seed, synth.T_WDOWN, 3, 0)
    qc, sc = cgen.weight_int8_grouped(key, 17, 9, sh.df, 128, synth.WEIGHT_SIGMA)
    qn, sn = quant.quantize_groupwise(synth.weight_f32(sh.seed, synth.T_WDOWN, 3, sh.d, sh.df, 17, 9))
    assert np.array_equal(qc, qn) and np.array_equal(sc.view(np.uint32), sn.view(np.uint32))


GSHAPE = synth.tiny_shape(L=3, dh=32, chan_unit=32, quant_group=32)


def _steps(sh, n):
    return synth.bf16_to_f32(synth.step_inputs_bf16(11, n, 1, sh.d)[:, 0])


@pytest.mark.parametrize("kind", ["groups", "qheads"])
def test_groupwise_mask_as_zero_equals_compacted(kind):
    from oracle import forward as fw
    from oracle import maskc
    sh = GSHAPE
    u = [[0, 3, 5], [2], [1, 4]]
    m = maskc.explicit(sh, [[0, 1], [1], [0]], u) if kind == "groups" else \
        maskc.explicit_qheads(sh, [[1, 2, 3], [3], [0, 2]], u)
    x = _steps(sh, 4).astype(np.float64)
    Xz = fw.decode(sh, m, x, 7, 7, dtype=np.float64)
    Xc = fw.decode(sh, m, x, 7, 7, compact=True, dtype=np.float64)
    assert np.linalg.norm(Xz - Xc) <= 1e-12 * np.linalg.norm(Xz)


def test_groupwise_panels_keep_the_scales_of_kept_groups():
    from oracle import pack, weights
    sh = GSHAPE
    lq = weights.gen_layer(sh, 1)
    assert lq.s["q"].shape == (sh.Hq * sh.dh, sh.d // 32) and lq.s["down"].shape == (sh.d, sh.df // 32)
    kc = list(range(64, 96)) + list(range(160, 192))  # channel units 2 and 5
    P = pack.pack_layer(sh, lq, [1], kc, [3])
    assert P["qkv_s"].shape == (3 * sh.dh, sh.d // 32)
    assert np.array_equal(P["o_s"], lq.s["o"][:, [3]])          # head 3 = column group 3
    assert np.array_equal(P["down_s"], lq.s["down"][:, [2, 5]])
    assert np.array_equal(P["gu_s"][0::2], lq.s["gate"][kc]) and np.array_equal(P["gu_s"][1::2], lq.s["up"][kc])
    # kept channels that split a scale group cannot be packed as whole groups
    with pytest.raises(ValueError):
        pack.pack_layer(sh, lq, [1], list(range(16, 48)), [3])


def test_groupwise_layer_is_closer_to_the_unquantized_layer():
    # one decode step of a layer on the unquantized FP32 weights against the same step on
    # per-row and on groupwise INT8 weights: the groupwise step is the closer one
    from oracle import forward as fw
    from oracle import weights
    row, grp = synth.tiny_shape(L=1, d=256, dh=64, df=512, chan_unit=64), \
        synth.tiny_shape(L=1, d=256, dh=64, df=512, chan_unit=64, quant_group=64)
    W0 = {}
    for name in weights.PROJ_NAMES:
        tid, r, c = weights.proj_dims(row, name)
        W0[name] = synth.weight_f32(row.seed, tid, 0, r, c).astype(np.float64)
    lq = weights.gen_layer(row, 0)
    W0["g_attn"], W0["g_mlp"] = lq.g_attn.astype(np.float64), lq.g_mlp.astype(np.float64)
    allg, allc = list(range(row.Hkv)), list(range(row.df))
    x = _steps(row, 1)[0].astype(np.float64)
    K, V = fw.prior_cache(row, 0, 7, 16, None, np.float64)
    y0, _, _ = fw.layer_step(row, W0, x, K, V, 16)
    errs = []
    for sh in (row, grp):
        W = weights.dense_zeroed(sh, weights.gen_layer(sh, 0), allg, allc, np.float64)
        y, _, _ = fw.layer_step(sh, W, x, K, V, 16)
        errs.append(np.linalg.norm(y - x - (y0 - x)) / np.linalg.norm(y0 - x))
    assert 0 < errs[1] < errs[0] < 5e-2
