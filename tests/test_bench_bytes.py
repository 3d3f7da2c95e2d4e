"""bench.py's algorithmic byte counts (the numerators of every reported roofline fraction)
against the oracle's packed panels: the INT8 rows and columns a plan streams per decode step,
for a whole-group mask and a query-head mask that keeps part of a group, plus the KV bytes."""
import dataclasses
import os
import sys

import pytest

import synth
from oracle import maskc, pack, weights

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402


def _expected(sh, pk, m_kv, c, m_q):
    """Per-launch bytes: panel weights (read once) + FP32 row scales + activations in / out."""
    d, dh = sh.d, sh.dh
    rows = pk["qkv_w"].shape[0]
    return {
        # weights, row scales, the input row and its norm gains, q out, K and V appended (BF16)
        "qkv": pk["qkv_w"].size + 4 * rows + 4 * d + 4 * d + 4 * m_q * dh + 2 * 2 * m_kv * dh,
        # weights, row scales, the attention output in, the residual read and written
        "o_proj": pk["o_w"].size + 4 * d + 4 * m_q * dh + 2 * 4 * d,
        # gate and up rows, their scales, the input row and gains, SiLU(gate) * up out
        "gate_up": pk["gu_w"].size + 4 * 2 * c + 4 * d + 4 * d + 4 * c,
        # weights, row scales, the hidden row in, the residual read and written
        "down": pk["down_w"].size + 4 * d + 4 * c + 2 * 4 * d,
    }


@pytest.mark.parametrize("kind", ["groups", "qheads"])
def test_gemv_bytes_count_the_packed_panels(kind):
    sh = synth.LAYER1  # g = 4, d_h = 64
    units = [list(range(0, sh.df, 2))]
    if kind == "groups":
        mask = maskc.explicit(sh, [[1]], units)
    else:  # group 0 keeps 3 of its 4 heads, group 1 keeps 2
        mask = maskc.explicit_qheads(sh, [[1, 2, 3, 4, 6]], units)
    qh = mask.qheads(sh, 0)
    pk = pack.pack_layer(sh, weights.gen_layer(sh, 0), mask.keep_groups[0], mask.keep_chans[0], qh)
    m_kv, c, m_q = len(mask.keep_groups[0]), len(mask.keep_chans[0]), len(qh)
    assert pk["qkv_w"].shape[0] == (m_q + 2 * m_kv) * sh.dh and pk["o_w"].shape[1] == m_q * sh.dh
    got = bench.gemv_bytes(sh, [(m_kv, c, m_q)])
    want = _expected(sh, pk, m_kv, c, m_q)
    for k, v in want.items():
        assert got[k] == v, (k, got[k], v)
    if kind == "groups":  # the two-entry form (kept groups, channels) means whole groups
        assert bench.gemv_bytes(sh, [(m_kv, c)]) == got


def test_grouped_store_adds_two_bytes_per_group_of_weights():
    sh = dataclasses.replace(synth.LAYER1, quant_group=64)
    dims = [(2, 704, 6)]
    per_row = bench.gemv_bytes(dataclasses.replace(sh, quant_group=0), dims)
    grouped = bench.gemv_bytes(sh, dims)
    d, dh, m_kv, c, m_q = sh.d, sh.dh, 2, 704, 6
    rows = (m_q + 2 * m_kv) * dh
    assert grouped["qkv"] - per_row["qkv"] == 2 * rows * (d // 64)
    assert grouped["o_proj"] - per_row["o_proj"] == 2 * d * (m_q * dh // 64)
    assert grouped["gate_up"] - per_row["gate_up"] == 2 * 2 * c * (d // 64)
    assert grouped["down"] - per_row["down"] == 2 * d * (c // 64)


def test_kv_bytes_read_the_kept_groups_and_append_one_position():
    dh, T = 128, 4101
    dims = [(5, 9000, 37), (8, 100), (0, 0, 0)]
    assert bench.kv_bytes(dims, dh, T) == (5 + 8) * (2 * T * dh * 2 + 2 * dh * 2)
