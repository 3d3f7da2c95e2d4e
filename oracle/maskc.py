"""Budgeted greedy construction of dependency-closed masks (Sec. 3.3). Test infrastructure only.

The paper's objective (Sec. 3.3): maximize sum_h M_h s_h subject to
sum_h c_h M_h <= B_t, solved greedily "by score per active FLOP" with the
dependency closure applied before each addition. Closure rules (Sec. 3.3):
a KV head stays whenever any of its query heads stays and query heads never
move across groups; a SwiGLU channel group keeps or drops its gate row, up
row and down column together.

Readings used here (the paper leaves them open):

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

Query-head candidates (``compile_mask_qheads``; Table 1 counts 64 per 70B
layer): a query head is charged its Q rows and O columns, and the closure
charges the K and V rows of its KV head to the first head of the group that is
accepted, so the ratio of a head is taken over its marginal cost at the moment
of the pick.

Pins: the single-layer closed form (1 of 2 groups and top-832 channels, ratio
0.569767...), agreement with a library sort (np.argsort) on the single-layer
case, the budget window, per-layer range, maximality of the result and
closure on every compiled mask. For query heads: hand-derived single-layer
cases (one where the closure cost reverses the order of two heads, one where a
second group does not fit, a ratio tie), two single-layer closed forms, the
reduction to the group compiler at g = 1, closure minimality and maximality
on the 8B/70B shapes.
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
    keep_groups: list  # per layer, sorted kept group (KV head) indices
    keep_units: list   # per layer, sorted kept channel-unit indices
    keep_chans: list   # per layer, sorted kept channel indices
    info: dict = field(default_factory=dict)
    keep_qheads: list | None = None  # per layer, sorted kept query heads; None = all g heads of each kept group

    def qheads(self, shape, layer: int) -> list:
        if self.keep_qheads is not None:
            return self.keep_qheads[layer]
        return [j * shape.g + i for j in self.keep_groups[layer] for i in range(shape.g)]


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
    if total > B:
        raise ValueError("the FLOP budget is below the forced minimum of one group and one channel unit per layer")
    groups = [[u for u in range(G) if acc[layer][u]] for layer in range(L)]
    units = [[u - G for u in range(G, G + U) if acc[layer][u]] for layer in range(L)]
    m = explicit(shape, groups, units)
    dense = ledger.dense_layer_flops(shape) * L
    m.info = dict(budget_flops=B, total_flops=total, dense_flops=dense, ratio=total / dense,
                  layer_budget=b, layer_cap=cap, layer_flops=lcost, layer_target_fixed=tt)
    return m


# --------------------------------------------------------------------------
# Query-head candidates with the GQA closure (Sec. 3.3; Table 1: 64 query-head
# candidates and 28 channel groups per 70B layer).
# --------------------------------------------------------------------------

def explicit_qheads(shape, qheads, units) -> Mask:
    """Mask from kept query heads and channel units; the kept KV heads are the closure
    (exactly the groups of the kept query heads)."""
    kq = [sorted(int(h) for h in hs) for hs in qheads]
    m = explicit(shape, [sorted({h // shape.g for h in hs}) for hs in kq], units)
    m.keep_qheads = kq
    return m


def compile_mask_qheads(shape, scores, target_u24, budget=0.57, r_lo=0.35, r_hi=0.85) -> Mask:
    """Greedy dependency-closed mask over query heads and channel units.

    ``scores`` [L, H_q + n_chan_units] (uint32): query heads first, then channel units.
    The candidate's cost is its marginal active FLOPs with the closure applied first
    (Sec. 3.3): a query head costs its Q rows and O columns, plus its KV head's K and
    V rows when no query head of its group is kept yet; a channel unit costs its
    gate/up rows and down columns. The greedy repeatedly accepts the candidate of
    highest score per marginal cost among those that still fit; costs change as KV
    heads come on, so the ratios are taken afresh at every pick. The phases, budgets
    and tie order are those of ``compile_mask`` (query head before channel unit, then
    lower index; globally lower layer first). With g = 1 a query head's marginal cost
    is always a whole group's and the result equals ``compile_mask``'s.
    """
    L, Hq, g, U = shape.L, shape.Hq, shape.g, shape.n_chan_units
    scores = np.asarray(scores, dtype=np.uint64)
    assert scores.shape == (L, Hq + U)
    c_q, c_kv, c_u = ledger.qhead_cost(shape), ledger.kv_cost(shape), ledger.chan_unit_cost(shape)
    b, cap, B, tt = _layer_budgets(shape, target_u24, budget, r_lo, r_hi)

    kept = [[False] * (Hq + U) for _ in range(L)]
    kv_on = [[False] * shape.Hkv for _ in range(L)]
    lcost = [0] * L

    def marginal(layer, u):
        if u < Hq:
            return c_q + (0 if kv_on[layer][u // g] else c_kv)
        return c_u

    def accept(layer, u):
        c = marginal(layer, u)
        kept[layer][u] = True
        if u < Hq:
            kv_on[layer][u // g] = True
        lcost[layer] += c
        return c

    def precedes(a, c, layer_first):
        # a, c = (layer, unit, marginal cost): higher score/cost first, then the tie order
        sa, sc = int(scores[a[0], a[1]]), int(scores[c[0], c[1]])
        lhs, rhs = sa * c[2], sc * a[2]
        if lhs != rhs:
            return lhs > rhs
        ka = (a[0], a[1] >= Hq, a[1]) if layer_first else (a[1] >= Hq, a[1], a[0])
        kc = (c[0], c[1] >= Hq, c[1]) if layer_first else (c[1] >= Hq, c[1], c[0])
        return ka < kc

    def best_fitting(layers, fits, layer_first):
        best = None
        for layer in layers:
            for u in range(Hq + U):
                if kept[layer][u]:
                    continue
                cand = (layer, u, marginal(layer, u))
                if fits(cand) and (best is None or precedes(cand, best, layer_first)):
                    best = cand
        return best

    for layer in range(L):
        # (1) forced minimum: best query head (with its KV head) and best channel unit
        for lo_u, hi_u in ((0, Hq), (Hq, Hq + U)):
            accept(layer, max(range(lo_u, hi_u), key=lambda u: (int(scores[layer, u]), -u)))
        # (2) per-layer greedy within the layer budget
        while True:
            cand = best_fitting([layer], lambda c: lcost[c[0]] + c[2] <= b[c[0]], False)
            if cand is None:
                break
            accept(layer, cand[1])
    # (3) global top-up within B and the per-layer cap
    total = sum(lcost)
    while True:
        cand = best_fitting(range(L), lambda c: total + c[2] <= B and lcost[c[0]] + c[2] <= cap[c[0]], True)
        if cand is None:
            break
        total += accept(cand[0], cand[1])
    if total > B:
        raise ValueError("the FLOP budget is below the forced minimum of one head and one channel unit per layer")
    qheads = [[u for u in range(Hq) if kept[layer][u]] for layer in range(L)]
    units = [[u - Hq for u in range(Hq, Hq + U) if kept[layer][u]] for layer in range(L)]
    m = explicit_qheads(shape, qheads, units)
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
        qh = mask.qheads(shape, layer)
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
