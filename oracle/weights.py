"""Regeneration and quantization of the synthetic dense model. Test infrastructure only.

Every dense projection is generated in PyTorch [out, in] layout from the
seeded recipe of ``synth`` (N(0, 0.02), FP32) and quantized per output row with
``oracle.quant`` (or, bit-identically, the oracle's C regenerator for large
layers); a shape with ``quant_group`` > 0 takes the groupwise format instead
(one BF16 scale per output row and run of ``quant_group`` input columns). The result is the shared INT8 store of the paper's backing-store
semantics (Appendix, "Backing-store semantics"): one copy of every projection,
independent of any mask.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

import synth
from . import cgen
from .quant import dequantize, quantize_groupwise, quantize_rows

# (tensor id, rows, cols) of each projection as functions of the shape
_PROJ = {
    "q": (synth.T_WQ, lambda s: s.Hq * s.dh, lambda s: s.d),
    "k": (synth.T_WK, lambda s: s.Hkv * s.dh, lambda s: s.d),
    "v": (synth.T_WV, lambda s: s.Hkv * s.dh, lambda s: s.d),
    "o": (synth.T_WO, lambda s: s.d, lambda s: s.Hq * s.dh),
    "gate": (synth.T_WGATE, lambda s: s.df, lambda s: s.d),
    "up": (synth.T_WUP, lambda s: s.df, lambda s: s.d),
    "down": (synth.T_WDOWN, lambda s: s.d, lambda s: s.df),
}
PROJ_NAMES = tuple(_PROJ)


@dataclass
class LayerQ:
    """Quantized dense layer: q[name] int8 [out, in], s[name] float32 [out] (or
    [out, in / group] for a groupwise store), norm gains."""
    q: dict
    s: dict
    g_attn: np.ndarray
    g_mlp: np.ndarray


def proj_dims(shape, name):
    tid, r, c = _PROJ[name]
    return tid, r(shape), c(shape)


def gen_proj_q(shape, layer: int, name: str, row0: int = 0, nrows: int | None = None,
               use_c: bool | None = None):
    """Quantized rows [row0, row0+nrows) of one projection: (q int8, s float32)."""
    tid, rows, cols = proj_dims(shape, name)
    if nrows is None:
        nrows = rows - row0
    if use_c is None:
        use_c = nrows * cols > (1 << 20) and cgen.available()
    key = synth.stream_key(shape.seed, tid, layer, 0)
    group = shape.quant_group
    if use_c:
        if group:
            return cgen.weight_int8_grouped(key, row0, nrows, cols, group, synth.WEIGHT_SIGMA)
        return cgen.weight_int8(key, row0, nrows, cols, synth.WEIGHT_SIGMA)
    w = synth.weight_f32(shape.seed, tid, layer, rows, cols, row0, nrows)
    return quantize_groupwise(w, group) if group else quantize_rows(w)


def gen_layer(shape, layer: int, use_c: bool | None = None) -> LayerQ:
    q, s = {}, {}
    for name in PROJ_NAMES:
        q[name], s[name] = gen_proj_q(shape, layer, name, use_c=use_c)
    return LayerQ(q, s, synth.gamma_f32(shape.seed, synth.T_GAMMA_ATTN, layer, shape.d),
                  synth.gamma_f32(shape.seed, synth.T_GAMMA_MLP, layer, shape.d))


def gamma_final(shape) -> np.ndarray:
    return synth.gamma_f32(shape.seed, synth.T_GAMMA_FINAL, 0, shape.d)


def lm_head_f32(shape, row0: int = 0, nrows: int | None = None) -> np.ndarray:
    return synth.bf16_to_f32(synth.lm_head_bf16(shape.seed, shape.vocab, shape.d, row0, nrows))


def dense_zeroed(shape, lq: LayerQ, keep_groups, keep_chans, dtype=np.float32, keep_qheads=None) -> dict:
    """Dequantized dense matrices with the pruned units set to zero (mask-as-zero).

    ``keep_qheads`` (sorted query heads) prunes single query heads: their Q rows and O
    columns are zeroed; K/V rows are zeroed for the groups not in ``keep_groups``. The
    default keeps all g query heads of every kept group.
    """
    g, dh = shape.g, shape.dh
    W = {name: dequantize(lq.q[name], lq.s[name], dtype) for name in PROJ_NAMES}
    kg = set(keep_groups)
    qh = set(keep_qheads) if keep_qheads is not None else {j * g + i for j in kg for i in range(g)}
    assert all(h // g in kg for h in qh), "a kept query head needs its KV head (GQA closure)"
    for h in range(shape.Hq):
        if h not in qh:
            W["q"][h * dh:(h + 1) * dh, :] = 0
            W["o"][:, h * dh:(h + 1) * dh] = 0
    for j in range(shape.Hkv):
        if j not in kg:
            W["k"][j * dh:(j + 1) * dh, :] = 0
            W["v"][j * dh:(j + 1) * dh, :] = 0
    keep_c = np.zeros(shape.df, dtype=bool)
    keep_c[np.asarray(keep_chans, dtype=np.int64)] = True
    W["gate"][~keep_c, :] = 0
    W["up"][~keep_c, :] = 0
    W["down"][:, ~keep_c] = 0
    W["g_attn"] = lq.g_attn.astype(dtype)
    W["g_mlp"] = lq.g_mlp.astype(dtype)
    return W
