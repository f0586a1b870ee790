"""MultiOSR: per-layer and per-linear OSR allocation (SDQ-LLM section 3.4).

The paper states the rule in prose only (section 3.4, Fig. 4): given a
target mean OSR, decoder layers are ranked by total weight variance and given
OSRs accordingly (lower variance -> more sensitive -> higher OSR); inside a
layer, the layer's OSR is spread over its linears inversely to their weight
variance and in proportion to their size.  This module makes that concrete
(the exact formula is ours; the paper gives none):

1. Layer targets: sort layers by total variance, ascending, and lay a linear
   ladder from ``mean + spread`` (lowest variance) down to ``mean - spread``
   (highest); for four equal layers at mean 2 and spread 1/2 the rungs are
   2.5, 2.17, 1.83, 1.5.
2. Within a layer: continuous target ``osr_i* proportional to size_i /
   variance_i``, normalised so the parameter-weighted mean equals the layer
   target.
3. In both steps the continuous targets become allowed values: the
   assignment closest to the targets (parameter-weighted squared distance)
   among those whose parameter-weighted mean is within ``tol`` of the
   target mean, by exhaustive search up to 2^16 assignments and, beyond, by single
   steps from the nearest values toward the mean, cheapest first (four equal
   layers at mean 2: 2.5, 2, 2, 1.5).

The allowed set is any list of OSRs with OSR * B an integer
(:func:`allowed_osrs`); the default is {1.5, 2, 2.5, 3}.  Host-side tool (no
GPU work); ``python -m paper_2510_03275_gb300.multiosr --config 3`` prints
the map of a workload as JSON.
"""
from __future__ import annotations

import argparse
import itertools
import json
from fractions import Fraction

ALLOWED = (Fraction(3, 2), Fraction(2), Fraction(5, 2), Fraction(3))
TOL = Fraction(1, 50)


def allowed_osrs(block: int, lo=Fraction(1), hi=Fraction(4), step=Fraction(1, 2)):
    """OSRs lo, lo + step, ..., hi with OSR * block an integer."""
    out, o = [], Fraction(lo)
    while o <= hi:
        if (o * block).denominator == 1:
            out.append(o)
        o += Fraction(step)
    return tuple(out)


def _weighted_mean(sizes, osrs):
    return sum(Fraction(s) * o for s, o in zip(sizes, osrs)) / sum(sizes)


def _nearest(allowed, x):
    return min(allowed, key=lambda a: (abs(float(a) - x), a))


def layer_targets(total_variances, mean=Fraction(2), sizes=None, allowed=ALLOWED, spread=Fraction(1, 2),
                  tol=TOL):
    """Per-layer OSR from the ranking of the layers' total variances."""
    n = len(total_variances)
    sizes = [1] * n if sizes is None else list(sizes)
    allowed = tuple(sorted(allowed))
    order = sorted(range(n), key=lambda i: total_variances[i])
    rung = [0.0] * n
    for rank, i in enumerate(order):
        frac = 0.0 if n == 1 else 1.0 - 2.0 * rank / (n - 1)
        rung[i] = float(mean) + float(spread) * frac
    return _fit_mean(sizes, rung, mean, allowed, tol)


def _fit_mean(sizes, want, mean, allowed, tol):
    """Allowed values close to ``want`` (parameter-weighted squared distance)
    with a weighted mean within ``tol`` of ``mean``: exhaustive search while
    there are at most 2^16 assignments; beyond, from the nearest values,
    single steps toward the mean that give the smallest distance increase per
    unit of mean corrected."""
    n = len(want)
    allowed = tuple(sorted(allowed))

    def cost(vals):
        return sum(s * (float(o) - w) ** 2 for s, o, w in zip(sizes, vals, want))

    if len(allowed) ** n <= 1 << 16:
        best, best_cost = None, None
        for combo in itertools.product(allowed, repeat=n):
            if abs(_weighted_mean(sizes, combo) - Fraction(mean)) > tol:
                continue
            c = cost(combo)
            if best_cost is None or c < best_cost - 1e-12:
                best, best_cost = list(combo), c
        if best is not None:
            return best
    out = [_nearest(allowed, w) for w in want]
    for _ in range(8 * n * len(allowed)):
        miss = _weighted_mean(sizes, out) - Fraction(mean)
        if abs(miss) <= tol:
            break
        step = -1 if miss > 0 else 1
        best, best_score = None, None
        for i in range(n):
            k = allowed.index(out[i]) + step
            if not 0 <= k < len(allowed):
                continue
            trial = out[:i] + [allowed[k]] + out[i + 1:]
            gain = abs(miss) - abs(_weighted_mean(sizes, trial) - Fraction(mean))
            if gain <= 0:
                continue
            score = (cost(trial) - cost(out)) / float(gain)
            if best_score is None or score < best_score:
                best, best_score = trial, score
        if best is None:
            break
        out = best
    return out


def within_layer(sizes, variances, target, allowed=ALLOWED, tol=TOL):
    """Per-linear OSRs of one layer (see the module docstring, step 2)."""
    prio = [s / v for s, v in zip(sizes, variances)]
    tot = sum(sizes)
    norm = sum(s * p for s, p in zip(sizes, prio)) / tot
    want = [float(target) * p / norm for p in prio]
    return _fit_mean(sizes, want, target, allowed, tol)


def allocate(sizes, variances, mean=Fraction(2), allowed=ALLOWED, spread=Fraction(1, 2), tol=TOL):
    """sizes, variances: per layer, per linear.  Returns OSRs per layer/linear."""
    totals = [sum(s * v for s, v in zip(sl, vl)) for sl, vl in zip(sizes, variances)]
    targets = layer_targets(totals, mean, [sum(sl) for sl in sizes], allowed, spread, tol)
    return [within_layer(sl, vl, t, allowed, tol) for sl, vl, t in zip(sizes, variances, targets)]


def allocate_from_weights(layers, mean=Fraction(2), **kw):
    """``layers``: per layer, a list of weight matrices (numpy arrays or
    torch tensors); sizes are element counts, variances the matrices'
    population variances."""
    sizes, variances = [], []
    for lay in layers:
        sizes.append([int(w.numel()) if hasattr(w, "numel") else int(w.size) for w in lay])
        variances.append([float(w.float().var(unbiased=False)) if hasattr(w, "numel") else float(w.var())
                          for w in lay])
    return allocate(sizes, variances, mean, **kw)


def summary(osrs, sizes):
    """Parameter-weighted mean OSR and the storage it implies: bits per
    original weight at 2 bits per code and in base-3 (1.6 bits per code),
    and eq. (14)'s compression ratio eta = N OSR / 16 at N = 1.58."""
    flat_o = [o for lay in osrs for o in lay]
    flat_s = [s for lay in sizes for s in lay]
    m = _weighted_mean(flat_s, flat_o)
    return {"mean_osr": float(m), "bits_per_weight_2bit": 2.0 * float(m),
            "bits_per_weight_base3": 1.6 * float(m), "eta_eq14": 1.58 * float(m) / 16.0}


def main(argv=None):
    from . import workloads as W
    ap = argparse.ArgumentParser(description="MultiOSR allocation of a synthetic workload (JSON)")
    ap.add_argument("--config", type=int, default=3)
    ap.add_argument("--mean", type=Fraction, default=Fraction(2))
    ap.add_argument("--allowed", default="3/2,2,5/2,3", help="comma-separated OSRs")
    ap.add_argument("--spread", type=Fraction, default=Fraction(1, 2))
    a = ap.parse_args(argv)
    allowed = tuple(Fraction(x) for x in a.allowed.split(","))
    cfg = W.config(a.config, multiosr=lambda sz, var: allocate(sz, var, a.mean, allowed, a.spread))
    per = {}
    for lin in cfg.linears:
        per[lin.name] = str(lin.osr)
    sizes = [[lin.n_out * lin.k_in for lin in cfg.linears]]
    out = {"workload": cfg.name, "osr": per, **summary([[lin.osr for lin in cfg.linears]], sizes)}
    print(json.dumps(out))
    return out


if __name__ == "__main__":
    main()
