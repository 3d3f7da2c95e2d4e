"""Active-FLOP ledger (Appendix, Eq. flop-attn and Eq. flop-mlp). Test infrastructure only.

Per decoder layer and token, with m_q / m_kv retained query / KV heads and c
retained SwiGLU channels:

    F_attn = 2 d d_h (m_q + 2 m_kv) + 2 d_h m_q d        (Q, K, V and O projections)
    F_mlp  = 6 d c                                       (gate, up, down)

The active-FLOP ratio is sum over layers of the retained FLOPs divided by the
same sum at full width; embeddings, final norm and LM head are excluded from
the budget (the paper states they are dense and enter both sides unchanged).
A KV head is charged once per retained group; with query-head candidates a
query head costs 2 d d_h (Q) + 2 d_h d (O) and a KV head 4 d d_h (K and V).

Pins: the closed forms of the three shapes (single layer 5,636,096 FLOP/layer,
8B 436,207,616, 70B 1,711,276,032), the 70B candidate count 80 x (64 + 28) =
7,360 (Table 1), and the "ratio from launched tile shapes" check of the
appendix's ledger table: FLOPs recounted from the packed panel shapes equal
the analytic ledger.
"""
from __future__ import annotations


def layer_flops(shape, m_q: int, m_kv: int, c: int) -> int:
    d, dh = shape.d, shape.dh
    f_attn = 2 * d * dh * (m_q + 2 * m_kv) + 2 * dh * m_q * d
    f_mlp = 6 * d * c
    return f_attn + f_mlp


def dense_layer_flops(shape) -> int:
    return layer_flops(shape, shape.Hq, shape.Hkv, shape.df)


def group_cost(shape) -> int:
    """Marginal FLOPs of one GQA group (a KV head with its g query heads)."""
    return layer_flops(shape, shape.g, 1, 0)


def qhead_cost(shape) -> int:
    """FLOPs of one query head alone (its Q rows and O columns; Sec. 3.3 query-head candidates)."""
    return layer_flops(shape, 1, 0, 0)


def kv_cost(shape) -> int:
    """FLOPs of one KV head (its K and V rows), charged by the closure with its first query head."""
    return layer_flops(shape, 0, 1, 0)


def chan_unit_cost(shape) -> int:
    """Marginal FLOPs of one SwiGLU channel unit (chan_unit coupled channels)."""
    return layer_flops(shape, 0, 0, shape.chan_unit)


def unit_costs(shape) -> list[int]:
    """Cost of each unit of a layer: H_kv groups first, then the channel units."""
    return [group_cost(shape)] * shape.Hkv + [chan_unit_cost(shape)] * shape.n_chan_units


def paper_candidate_count(shape) -> int:
    """Candidates as the paper counts them: one per query head and per 1,024-channel group."""
    return shape.L * (shape.Hq + shape.df // 1024)


def mask_flops(shape, keep_groups, keep_chans, keep_qheads=None) -> int:
    """Retained layer FLOPs of a mask; ``keep_qheads`` (per layer) overrides the g query
    heads per kept group of a group-granular mask."""
    if keep_qheads is None:
        keep_qheads = [[0] * (shape.g * len(kg)) for kg in keep_groups]
    return sum(layer_flops(shape, len(qh), len(kg), len(kc))
               for kg, kc, qh in zip(keep_groups, keep_chans, keep_qheads))


def mask_ratio(shape, keep_groups, keep_chans, keep_qheads=None) -> float:
    return mask_flops(shape, keep_groups, keep_chans, keep_qheads) / (shape.L * dense_layer_flops(shape))


def launched_flops(panels_per_layer) -> int:
    """2 x rows x cols summed over every packed projection panel (one MAC = 2 FLOPs)."""
    tot = 0
    for p in panels_per_layer:
        for name in ("qkv", "o", "gu", "down"):
            r, c = p[name + "_w"].shape
            tot += 2 * r * c
    return tot
