"""Pins of the oracle's quantizer and active-FLOP ledger."""
import os

import numpy as np

import synth
from oracle import cgen, ledger, maskc, pack, quant, weights

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def test_quant_hand_cases():
    # max |w| = 127 -> s = 1 exactly; ties round half to even
    w = np.array([[127.0, 2.5, 3.5, -2.5, 0.5, -127.0, 1.49]], dtype=np.float32)
    q, s = quant.quantize_rows(w)
    assert s[0] == np.float32(1.0)
    assert q.tolist() == [[127, 2, 4, -2, 0, -127, 1]]


def test_quant_zero_row_and_symmetry():
    w = np.zeros((2, 8), dtype=np.float32)
    w[1] = np.linspace(-0.3, 0.2, 8, dtype=np.float32)
    q, s = quant.quantize_rows(w)
    assert s[0] == 0 and not q[0].any()
    qn, sn = quant.quantize_rows(-w)
    assert np.array_equal(qn, -q) and np.array_equal(sn, s)
    # the row maximum maps to +-127
    assert np.abs(q[1]).max() == 127


def test_quant_error_bound():
    rng = np.random.default_rng(1)
    w = (rng.standard_normal((64, 1000)) * 0.02).astype(np.float32)
    q, s = quant.quantize_rows(w)
    err = np.abs(quant.dequantize_rows(q, s, np.float64) - w.astype(np.float64))
    assert np.all(err <= s.astype(np.float64)[:, None] * (0.5 + 1e-6))
    assert np.abs(q).max() <= 127


def test_quant_numpy_equals_c():
    rng = np.random.default_rng(2)
    w = (rng.standard_normal((16, 777)) * 0.02).astype(np.float32)
    q, s = quant.quantize_rows(w)
    for r in range(16):
        qc, sc = cgen.quant_row(w[r])
        assert np.array_equal(qc, q[r]) and np.float32(sc) == s[r]


def test_layer_regeneration_c_equals_numpy():
    sh = synth.tiny_shape(d=256, df=384)
    for name in ("q", "down", "gate"):
        a = weights.gen_proj_q(sh, 1, name, use_c=True)
        b = weights.gen_proj_q(sh, 1, name, use_c=False)
        assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
    # a row window equals the same rows of the whole matrix
    qa, sa = weights.gen_proj_q(sh, 0, "up", row0=17, nrows=5, use_c=True)
    qb, sb = weights.gen_proj_q(sh, 0, "up", use_c=False)
    assert np.array_equal(qa, qb[17:22]) and np.array_equal(sa, sb[17:22])


def _closed_forms():
    rows = {}
    with open(os.path.join(GOLD, "flop_ledger_closed_forms.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            parts = line.split()
            rows[parts[0]] = parts[1:]
    return rows


def test_ledger_closed_forms():
    g = _closed_forms()
    for name, sh in (("layer1", synth.LAYER1), ("llama3_8b", synth.LLAMA3_8B), ("llama3_70b", synth.LLAMA3_70B)):
        dense, gc, cc, cand = g[name]
        assert ledger.dense_layer_flops(sh) == int(dense)
        assert ledger.group_cost(sh) == int(gc)
        assert ledger.chan_unit_cost(sh) == int(cc)
        if cand != "-":
            assert ledger.paper_candidate_count(sh) == int(cand)
        # groups and channel units partition the dense layer exactly
        assert sh.Hkv * ledger.group_cost(sh) + sh.n_chan_units * ledger.chan_unit_cost(sh) == int(dense)


def test_ledger_equals_launched_panel_shapes():
    # The appendix's check: FLOPs recounted from the dimensions actually packed
    sh = synth.tiny_shape()
    sc = synth.mask_scores_u32(77, sh.L, sh.n_units)
    m = maskc.compile_mask(sh, sc, synth.layer_target_u24(77, sh.L))
    panels = [pack.pack_layer(sh, weights.gen_layer(sh, l), m.keep_groups[l], m.keep_chans[l]) for l in range(sh.L)]
    assert ledger.launched_flops(panels) == ledger.mask_flops(sh, m.keep_groups, m.keep_chans)
    full = maskc.all_keep(sh)
    panels = [pack.pack_layer(sh, weights.gen_layer(sh, l), full.keep_groups[l], full.keep_chans[l]) for l in range(sh.L)]
    assert ledger.launched_flops(panels) == sh.L * ledger.dense_layer_flops(sh)
