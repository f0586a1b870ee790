"""CPU: the MultiOSR allocation helper (section 3.4, prose only) against the
properties the prose and the harness rule fix: lower-variance layers get
higher OSR, every OSR is one of the allowed values, each layer's
parameter-weighted mean OSR is within +-0.02 of its target, the stack's mean
is 2.0 +-0.02, and inside a layer a lower-variance linear of the same size
never gets a lower OSR.  (The exact formula is this package's own reading;
its parity with the paper stays unpinned.)"""
from fractions import Fraction

import numpy as np
import pytest

from paper_2510_03275_gb300 import multiosr as MO
from paper_2510_03275_gb300 import workloads as W


def test_layer_ladder_follows_variance():
    tv = [3.0, 1.0, 4.0, 2.0]
    t = MO.layer_targets(tv)
    assert t == [Fraction(2), Fraction(5, 2), Fraction(3, 2), Fraction(2)]
    assert sum(t) / len(t) == 2
    for perm in ([1, 0, 3, 2], [3, 2, 1, 0]):
        tp = MO.layer_targets([tv[i] for i in perm])
        assert tp == [t[i] for i in perm]


@pytest.mark.parametrize("seed", range(6))
def test_within_layer_mean_and_allowed_set(seed):
    rng = np.random.default_rng(seed)
    sizes = [int(s) for s in rng.integers(1, 8, size=5) * 1_000_000]
    variances = list(rng.uniform(0.5, 2.0, size=5))
    for target in (Fraction(3, 2), Fraction(2), Fraction(5, 2)):
        o = MO.within_layer(sizes, variances, target)
        assert all(x in MO.ALLOWED for x in o)
        mean = Fraction(sum(s * x for s, x in zip(sizes, o)), sum(sizes))
        assert abs(mean - target) <= Fraction(1, 50)


def test_within_layer_lower_variance_never_lower_osr():
    sizes = [4_000_000] * 4
    variances = [0.5, 1.0, 2.0, 4.0]
    o = MO.within_layer(sizes, variances, Fraction(2))
    assert all(a >= b for a, b in zip(o, o[1:]))
    assert o[0] > o[-1]


def test_llama13b_stack_mean_osr():
    """The 4-layer LLaMA-13B stack of the benchmark workloads: the overall
    parameter-weighted mean OSR is 2.0 +-0.02, with every layer at its
    ladder target within +-0.02."""
    cfg = W.config(3, multiosr=MO.allocate)
    lins = cfg.linears
    tot = sum(l.n_out * l.k_in for l in lins)
    mean = sum(Fraction(l.osr) * l.n_out * l.k_in for l in lins) / tot
    assert abs(mean - 2) <= Fraction(1, 50)
    assert {Fraction(l.osr) for l in lins} <= set(MO.ALLOWED)
