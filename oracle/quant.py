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
the oracle's C quantizer (oracle/csrc/ogen.c).
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
    return (q.astype(dtype) * np.asarray(s, dtype=dtype)[:, None]).astype(dtype)
