"""Per-turn plan choice with the dense fallback (Sec. 3.3; Table 1: tau = 0.85). Test
infrastructure only.

Given the router's task distribution p(t | x) over the task masks, the turn runs the sparse
plan of the most probable task when that probability reaches tau, and the dense plan
otherwise. Readings: ties go to the lower task index; the dense plan is numbered after the
task masks (index n for n masks); a probability exactly equal to tau dispatches the sparse
plan (the paper falls back only when the maximum is below tau).

Pins: hand cases of the rule at tau = 0.85, the tie order, and agreement with numpy's argmax
on random distributions.
"""
from __future__ import annotations

import numpy as np


def choose_plan(probs, tau: float = 0.85) -> int:
    p = [float(v) for v in probs]
    if not p or any(not np.isfinite(v) or v < 0 for v in p) or not 0.0 <= tau <= 1.0:
        raise ValueError("need finite non-negative probabilities and tau in [0, 1]")
    best = 0
    for i in range(1, len(p)):
        if p[i] > p[best]:
            best = i
    return best if p[best] >= tau else len(p)
