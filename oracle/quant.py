"""Per-output-channel symmetric INT8 quantizer (numpy). Test infrastructure only.

The paper packs "symmetric ... INT8 weights" with fused dequantization
(Sec. 4, Table 1). The build's reading quantizes each OUTPUT row of a PyTorch
[out, in] matrix with one FP32 scale (the paper's group size 128 with BF16
scales is a later variant):

    a = max_j |w_j|,  s = fl32(a / 127),  q_j = clamp(rint(fl32(w_j / s)), -127, 127)

rint is round-half-to-even; a row of zeros gets s = 0 and q = 0. Scales depend
only on the dense row, never on a mask, so a compacted panel carries the same
scale as the dense row it came from.

Pins: hand cases (a row whose maximum is 127*s maps to +-127, zero rows, ties
to even), the elementwise error bound |s*q - w| <= s/2, and bit equality with
the oracle's C quantizer (oracle/csrc/ogen.c). The groupwise variant below is
pinned by the same kinds of hand cases, its own error bound, a single-group
matrix against the per-row rule with a BF16 scale, and BF16 rounding checked
against exact ties and torch's bfloat16 conversion.
"""
from __future__ import annotations

import numpy as np


def quantize_rows(w: np.ndarray):
    """w: float32 [rows, cols] -> (q int8 [rows, cols], s float32 [rows])."""
    w = np.asarray(w, dtype=np.float32)
    a = np.max(np.abs(w), axis=1)
    s = (a / np.float32(127.0)).astype(np.float32)
    safe = np.where(s == 0, np.float32(1.0), s).astype(np.float32)
    r = np.rint((w / safe[:, None]).astype(np.float32))
    r = np.clip(r, -127, 127)
    r[s == 0, :] = 0
    return r.astype(np.int8), s


def dequantize_rows(q: np.ndarray, s: np.ndarray, dtype=np.float32) -> np.ndarray:
    """W~ = s * Q per output row."""
    w = q.astype(dtype)
    np.multiply(w, np.asarray(s, dtype=dtype)[:, None], out=w)  # in place: one product per element
    return w


# ------------------------------------------------------------------ groupwise variant
# The paper's own deployment format (Table 1 "Symmetric groupwise INT8 weights, group size
# 128; ... BF16 scales"; Appendix "Backing-store semantics"): each output row is cut into
# groups of 128 consecutive input columns, each group with its own scale stored in BF16. The
# paper gives no formula; the reading here keeps the per-row rule above per group, with the
# scale rounded to BF16 before it divides:
#
#     a = max_{j in g} |w_j|,  s = bf16(fl32(a / 127)),  q_j = clamp(rint(fl32(w_j / s)), -127, 127)
#
# bf16() is round-to-nearest-even on the FP32 bit pattern. Rounding the scale down can push
# |w_j / s| just past 127; the clamp absorbs it. A group of zeros gets s = 0 and q = 0.

def to_bf16(x: np.ndarray) -> np.ndarray:
    """FP32 -> nearest BF16 value (ties to even), returned as FP32 (finite inputs)."""
    u = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    r = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return (r << 16).astype(np.uint32).view(np.float32)


def quantize_groupwise(w: np.ndarray, group: int = 128):
    """w: float32 [rows, cols] (cols a multiple of group) ->
    (q int8 [rows, cols], s float32 [rows, cols // group], every s a BF16 value)."""
    w = np.asarray(w, dtype=np.float32)
    rows, cols = w.shape
    if cols % group:
        raise ValueError("columns must be a multiple of the group size")
    wg = w.reshape(rows, cols // group, group)
    a = np.max(np.abs(wg), axis=2)
    s = to_bf16((a / np.float32(127.0)).astype(np.float32))
    safe = np.where(s == 0, np.float32(1.0), s).astype(np.float32)
    r = np.rint((wg / safe[:, :, None]).astype(np.float32))
    r = np.clip(r, -127, 127)
    r[s == 0] = 0
    return r.reshape(rows, cols).astype(np.int8), s


def dequantize_groupwise(q: np.ndarray, s: np.ndarray, group: int = 128, dtype=np.float32) -> np.ndarray:
    """W~ = s_g * Q per (row, group of `group` columns)."""
    rows, cols = q.shape
    qg = q.reshape(rows, cols // group, group).astype(dtype)
    return (qg * np.asarray(s, dtype=dtype)[:, :, None]).reshape(rows, cols).astype(dtype)


def dequantize(q: np.ndarray, s: np.ndarray, dtype=np.float32) -> np.ndarray:
    """Per-row (s [rows]) or groupwise (s [rows, cols / group]) dequantization."""
    s = np.asarray(s)
    if s.ndim == 1:
        return dequantize_rows(q, s, dtype)
    if q.shape[1] == 0:
        return np.zeros(q.shape, dtype)
    return dequantize_groupwise(q, s, q.shape[1] // s.shape[1], dtype)
