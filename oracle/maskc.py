"""Budgeted greedy construction of dependency-closed masks (Sec. 3.3). Test infrastructure only.

The paper's objective (Sec. 3.3): maximize sum_h M_h s_h subject to
sum_h c_h M_h <= B_t, solved greedily "by score per active FLOP" with the
dependency closure applied before each addition. Closure rules (Sec. 3.3):
a KV head stays whenever any of its query heads stays and query heads never
move across groups; a SwiGLU channel group keeps or drops its gate row, up
row and down column together.

Readings used here (the paper leaves them open; all are listed in the design doc):

* Unit = a whole GQA group (KV head + its g query heads) or a block of
  ``chan_unit`` channels. Closure is then satisfied by construction and is
  still checked by ``closure_holds``.
* Scores are uint32 stand-ins for the predictor output s_h, ratio = s / c.
  Ratios are compared exactly by cross multiplication (integers), ties go to
  group before channel unit, then lower index (then lower layer globally).
* Per-layer retention targets t_l = LO + (HI-LO) * u24_l / 2**24 in fixed point
  2**-24 (LO, HI = the retention range), shifted by one common integer delta,
  the largest for which sum_l clamp(t_l + delta, LO, HI) * F_l <= T * sum_l F_l
  (T = budget in fixed point): the layer budget is b_l = floor(clamp(...) F_l / 2**24).
* Greedy: (1) every layer keeps its best group and best channel unit; (2) per
  layer, units in descending ratio are accepted while the layer stays within
  b_l (skip and continue); (3) a global top-up in descending ratio accepts a
  unit while the total stays within B = floor(T sum F / 2**24) and its layer
  within floor(HI F_l / 2**24).

Pins: the single-layer closed form (1 of 2 groups and top-832 channels, ratio
0.569767...), agreement with a library sort (np.argsort) on the single-layer
case, the budget window, per-layer range, maximality of the result and
closure on every compiled mask.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from functools import cmp_to_key

import numpy as np

from . import ledger

FIX_BITS = 24
FIX = 1 << FIX_BITS


def to_fixed(r: float) -> int:
    """Round a ratio to fixed point 2**-24 (floor(r * 2**24 + 0.5), exact in double)."""
    return int(math.floor(r * FIX + 0.5))


@dataclass
class Mask:
    keep_groups: list  # per layer, sorted kept group indices
    keep_units: list   # per layer, sorted kept channel-unit indices
    keep_chans: list   # per layer, sorted kept channel indices
    info: dict = field(default_factory=dict)


def all_keep(shape) -> Mask:
    return explicit(shape, [list(range(shape.Hkv))] * shape.L, [list(range(shape.n_chan_units))] * shape.L)


def explicit(shape, groups, units) -> Mask:
    kg = [sorted(int(j) for j in g) for g in groups]
    ku = [sorted(int(u) for u in us) for us in units]
    kc = [[u * shape.chan_unit + i for u in us for i in range(shape.chan_unit)] for us in ku]
    return Mask(kg, ku, kc)


def _layer_budgets(shape, target_u24, budget, r_lo, r_hi):
    L = shape.L
    T, LO, HI = to_fixed(budget), to_fixed(r_lo), to_fixed(r_hi)
    F = [ledger.dense_layer_flops(shape)] * L
    t = [LO + (((HI - LO) * int(target_u24[layer])) >> FIX_BITS) for layer in range(L)]
    b_fix = T * sum(F)

    def filled(delta):
        return sum(min(max(t[layer] + delta, LO), HI) * F[layer] for layer in range(L))

    lo, hi = -FIX, FIX  # filled(lo) <= b_fix requires LO <= T
    if filled(hi) <= b_fix:
        delta = hi
    else:
        while hi - lo > 1:  # invariant: filled(lo) <= b_fix < filled(hi)
            mid = (lo + hi) // 2
            if filled(mid) <= b_fix:
                lo = mid
            else:
                hi = mid
        delta = lo
    tt = [min(max(t[layer] + delta, LO), HI) for layer in range(L)]
    b = [(tt[layer] * F[layer]) >> FIX_BITS for layer in range(L)]
    cap = [(HI * F[layer]) >> FIX_BITS for layer in range(L)]
    B = b_fix >> FIX_BITS
    return b, cap, B, tt


def compile_mask(shape, scores, target_u24, budget=0.57, r_lo=0.35, r_hi=0.85) -> Mask:
    """Greedy dependency-closed mask from scores [L, H_kv + n_chan_units] (uint32)."""
    L, G, U = shape.L, shape.Hkv, shape.n_chan_units
    scores = np.asarray(scores, dtype=np.uint64)
    assert scores.shape == (L, G + U)
    cost = ledger.unit_costs(shape)
    b, cap, B, tt = _layer_budgets(shape, target_u24, budget, r_lo, r_hi)

    def kind(u):
        return 0 if u < G else 1

    def by_ratio(a, c):
        # a, c: (layer, unit); descending score/cost, then group<channel, lower index, lower layer
        sa, sc = int(scores[a[0], a[1]]), int(scores[c[0], c[1]])
        lhs, rhs = sa * cost[c[1]], sc * cost[a[1]]
        if lhs != rhs:
            return -1 if lhs > rhs else 1
        ka, kc = (kind(a[1]), a[1], a[0]), (kind(c[1]), c[1], c[0])
        return -1 if ka < kc else (1 if ka > kc else 0)

    def global_order(a, c):
        sa, sc = int(scores[a[0], a[1]]), int(scores[c[0], c[1]])
        lhs, rhs = sa * cost[c[1]], sc * cost[a[1]]
        if lhs != rhs:
            return -1 if lhs > rhs else 1
        ka, kc = (a[0], kind(a[1]), a[1]), (c[0], kind(c[1]), c[1])
        return -1 if ka < kc else (1 if ka > kc else 0)

    acc = [[False] * (G + U) for _ in range(L)]
    lcost = [0] * L
    for layer in range(L):
        # (1) forced minimum: best group and best channel unit (ties to lower index)
        for lo_u, hi_u in ((0, G), (G, G + U)):
            best = max(range(lo_u, hi_u), key=lambda u: (int(scores[layer, u]), -u))
            acc[layer][best] = True
            lcost[layer] += cost[best]
        # (2) per-layer walk in ratio order
        order = sorted(((layer, u) for u in range(G + U)), key=cmp_to_key(by_ratio))
        for _, u in order:
            if not acc[layer][u] and lcost[layer] + cost[u] <= b[layer]:
                acc[layer][u] = True
                lcost[layer] += cost[u]
    total = sum(lcost)
    # (3) global top-up
    rest = [(layer, u) for layer in range(L) for u in range(G + U) if not acc[layer][u]]
    rest.sort(key=cmp_to_key(global_order))
    for layer, u in rest:
        if total + cost[u] <= B and lcost[layer] + cost[u] <= cap[layer]:
            acc[layer][u] = True
            lcost[layer] += cost[u]
            total += cost[u]
    groups = [[u for u in range(G) if acc[layer][u]] for layer in range(L)]
    units = [[u - G for u in range(G, G + U) if acc[layer][u]] for layer in range(L)]
    m = explicit(shape, groups, units)
    dense = ledger.dense_layer_flops(shape) * L
    m.info = dict(budget_flops=B, total_flops=total, dense_flops=dense, ratio=total / dense,
                  layer_budget=b, layer_cap=cap, layer_flops=lcost, layer_target_fixed=tt)
    return m


# --------------------------------------------------------------------------
# Dependency closure at the level of individual matrices (Sec. 3.3).
# --------------------------------------------------------------------------

def expand(shape, mask: Mask) -> list[dict]:
    """Per-layer retained index sets of every projection implied by a mask."""
    out = []
    for layer in range(shape.L):
        kg, kc = mask.keep_groups[layer], mask.keep_chans[layer]
        qh = [j * shape.g + i for j in kg for i in range(shape.g)]
        out.append(dict(q_heads=set(qh), kv_heads=set(kg), o_heads=set(qh),
                        gate=set(kc), up=set(kc), down=set(kc)))
    return out


def closure_holds(shape, per_layer_sets) -> bool:
    """GQA rule: every kept query head's KV head is kept and O keeps exactly the kept
    query heads' columns; SwiGLU rule: gate rows, up rows and down columns agree."""
    for s in per_layer_sets:
        for h in s["q_heads"]:
            if h // shape.g not in s["kv_heads"]:
                return False
        if s["o_heads"] != s["q_heads"]:
            return False
        if not (s["gate"] == s["up"] == s["down"]):
            return False
    return True
