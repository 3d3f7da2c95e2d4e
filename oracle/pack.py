"""Packing of retained units into contiguous INT8 panels (Sec. 3.3, Appendix
"Backing-store semantics"). Test infrastructure only.

The paper packs each mask's retained heads and channels into contiguous
tensors over one shared INT8 store. The panel layout the build uses (and
which the library's panels must match byte for byte) is:

* ``qkv``  [(m_q + 2 m_kv) d_h, d]: for each kept group j in ascending order,
  the d_h rows of each of its kept query heads (of heads j g .. j g + g - 1, all g
  of them for a group-granular mask, ascending), then the d_h rows of K head j,
  then the d_h rows of V head j.
* ``o``    [d, m_q d_h]: the O-projection columns of the kept query heads in
  ascending head order; scales are the dense per-row scales [d].
* ``gu``   [2 c, d]: for each kept channel c_i in ascending order, the gate
  row c_i then the up row c_i.
* ``down`` [d, c]: the down-projection columns of the kept channels; scales
  are the dense per-row scales [d].

The all-keep mask packs to the shared store itself. In a groupwise store the
qkv / gu scale rows travel with their weight rows, and O / down keep the
scale columns of the kept column groups (kept heads and channel units must
then be whole scale groups: d_h and the channel unit multiples of the group).

Pin: the compacted forward (oracle.forward, ``compact=True``) consumes these
panels and must equal the mask-as-zero forward; a permuted or misaligned
panel fails that test.
"""
from __future__ import annotations

import numpy as np


def kept_qheads(shape, keep_groups, keep_qheads=None):
    """Kept query heads in ascending order (all g heads of each kept group by default)."""
    if keep_qheads is None:
        return [h for j in keep_groups for h in range(j * shape.g, (j + 1) * shape.g)]
    return sorted(keep_qheads)


def qkv_rows(shape, keep_groups, keep_qheads=None):
    """Dense-matrix row sources of the qkv panel: list of (proj, row)."""
    rows = []
    g, dh = shape.g, shape.dh
    qh = set(kept_qheads(shape, keep_groups, keep_qheads))
    for j in keep_groups:
        for h in range(j * g, (j + 1) * g):
            if h in qh:
                rows += [("q", h * dh + i) for i in range(dh)]
        rows += [("k", j * dh + i) for i in range(dh)]
        rows += [("v", j * dh + i) for i in range(dh)]
    return rows


def _column_groups(cols, group):
    """Scale groups of kept columns that come in whole runs of ``group``; else ValueError."""
    cols = np.asarray(cols, dtype=np.int64)
    if len(cols) % group or np.any(cols.reshape(-1, group) != cols[::group, None] + np.arange(group)) \
            or np.any(cols[::group] % group):
        raise ValueError("a groupwise store packs kept columns in whole scale groups only")
    return cols[::group] // group


def pack_layer(shape, lq, keep_groups, keep_chans, keep_qheads=None) -> dict:
    dh, grp = shape.dh, shape.quant_group
    srow = (shape.d // grp,) if grp else ()  # trailing scale dims of a row of the qkv / gu panels
    src = qkv_rows(shape, keep_groups, keep_qheads)
    qkv_w = np.stack([lq.q[p][r] for p, r in src]) if src else np.zeros((0, shape.d), np.int8)
    qkv_s = np.array([lq.s[p][r] for p, r in src], dtype=np.float32).reshape((len(src),) + srow)
    ocols = [h * dh + i for h in kept_qheads(shape, keep_groups, keep_qheads) for i in range(dh)]
    o_w = np.ascontiguousarray(lq.q["o"][:, ocols])
    kc = np.asarray(keep_chans, dtype=np.int64)
    gu_w = np.empty((2 * len(kc), shape.d), dtype=np.int8)
    gu_w[0::2] = lq.q["gate"][kc]
    gu_w[1::2] = lq.q["up"][kc]
    gu_s = np.empty((2 * len(kc),) + srow, dtype=np.float32)
    gu_s[0::2] = lq.s["gate"][kc]
    gu_s[1::2] = lq.s["up"][kc]
    down_w = np.ascontiguousarray(lq.q["down"][:, kc])
    if grp:  # O / down keep the scales of the kept column groups
        o_s = np.ascontiguousarray(lq.s["o"][:, _column_groups(ocols, grp)])
        down_s = np.ascontiguousarray(lq.s["down"][:, _column_groups(kc, grp)])
    else:
        o_s, down_s = lq.s["o"].copy(), lq.s["down"].copy()
    return dict(qkv_w=qkv_w, qkv_s=qkv_s, o_w=o_w, o_s=o_s, gu_w=gu_w, gu_s=gu_s,
                down_w=down_w, down_s=down_s)
