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


def test_llama13b_map_is_stable():
    """The allocation the 13B stack's tests and bench use (regression of the
    module's own output, not a paper value)."""
    cfg = W.config(3, multiosr=MO.allocate)
    got = [str(l.osr) for l in cfg.linears]
    assert got == ['3/2', '3/2', '3/2', '2', '3/2', '2', '3', '3/2', '2', '3/2', '3/2', '3', '3/2', '2',
                   '2', '3/2', '2', '3', '3', '3', '2', '3/2', '3/2', '3/2', '3/2', '3/2', '3/2', '3/2']


def test_allowed_osrs_respect_block():
    assert MO.allowed_osrs(128) == tuple(Fraction(k, 2) for k in range(2, 9))
    a = MO.allowed_osrs(4, step=Fraction(1, 8))
    assert all((o * 4).denominator == 1 for o in a) and Fraction(5, 4) in a and Fraction(9, 8) not in a


@pytest.mark.parametrize("n,mean", [(80, Fraction(2)), (32, Fraction(5, 2)), (7, Fraction(3, 2))])
def test_layer_targets_many_layers(n, mean):
    rng = np.random.default_rng(n)
    tv = list(rng.uniform(0.5, 3.0, size=n))
    allowed = MO.allowed_osrs(128, Fraction(1), Fraction(4))
    t = MO.layer_targets(tv, mean, allowed=allowed)
    assert all(o in allowed for o in t)
    assert abs(sum(t) / n - mean) <= MO.TOL
    order = np.argsort(tv)
    ranked = [t[i] for i in order]
    assert all(a >= b for a, b in zip(ranked, ranked[1:]))     # lower variance, no lower OSR
    assert ranked[0] > ranked[-1]


def test_layer_targets_weighted_by_size():
    sizes = [1, 1, 1, 9]
    t = MO.layer_targets([1.0, 2.0, 3.0, 4.0], Fraction(2), sizes)
    mean = sum(s * o for s, o in zip(sizes, t)) / sum(sizes)
    assert abs(mean - 2) <= MO.TOL


def test_within_layer_many_linears_greedy():
    rng = np.random.default_rng(3)
    sizes = [int(s) for s in rng.integers(1, 9, size=12) * 1_000_000]
    variances = list(rng.uniform(0.5, 2.0, size=12))
    o = MO.within_layer(sizes, variances, Fraction(2))
    mean = Fraction(sum(s * x for s, x in zip(sizes, o)), sum(sizes))
    assert abs(mean - 2) <= MO.TOL and all(x in MO.ALLOWED for x in o)


def test_allocate_from_weights_and_summary():
    rng = np.random.default_rng(0)
    layers = [[rng.standard_normal((64, 32)) * s for s in (0.01, 0.02, 0.04)] for _ in range(4)]
    osrs = MO.allocate_from_weights(layers)
    assert len(osrs) == 4 and all(len(l) == 3 for l in osrs)
    sizes = [[w.size for w in lay] for lay in layers]
    sm = MO.summary(osrs, sizes)
    assert abs(sm["mean_osr"] - 2.0) <= 0.02 + 1e-9
    assert abs(sm["bits_per_weight_base3"] - 1.6 * sm["mean_osr"]) < 1e-12
    # inside each layer the lowest-variance linear gets the highest OSR
    assert all(l[0] >= l[-1] for l in osrs)


def test_cli_prints_the_map(capsys):
    out = MO.main(["--config", "3"])
    assert len(out["osr"]) == 28 and abs(out["mean_osr"] - 2.0) <= 0.02
    assert '"workload": "llama-13b-4layers"' in capsys.readouterr().out


def test_shared_input_groups():
    g4 = [(n, [l.name for l in ms]) for n, ms in W.shared_input_groups(W.config(4))]
    assert g4 == [("qkv", ["q", "k", "v"]), ("o", ["o"]), ("gate_up", ["gate", "up"]), ("down", ["down"])]
    g1 = [n for n, _ in W.shared_input_groups(W.config(1))]
    assert g1 == ["qkv", "o", "fc1", "fc2"]
    # under MultiOSR, members with different OSRs stay separate plans
    g3 = W.shared_input_groups(W.config(3, multiosr=MO.allocate))
    assert all(len({l.osr for l in ms}) == 1 for _, ms in g3)
    assert sum(len(ms) for _, ms in g3) == 28
