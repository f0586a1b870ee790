"""CPU: the error bounds the GPU parity tests apply (tests/errbound.py)
against an fp64 emulation of each path's arithmetic, and against planted
mistakes in that emulation: the bounds must hold for the arithmetic as
described and fail for a term too few, a flipped sign or a wrong scale."""
import numpy as np
import pytest

import errbound as EB
import oracle as O
from paper_2510_03275_gb300 import workloads as W

E2M1 = np.array([0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0])


def _e2m1(v):
    """Round to the nearest e2m1 value (ties to the even code)."""
    a = np.abs(v)
    d = np.abs(a[..., None] - E2M1)
    best = d.min(axis=-1, keepdims=True)
    idx = np.where(np.isclose(d, best, rtol=0, atol=0), np.arange(8), 99)
    ties = (idx % 2 == 0) & (idx < 99)
    pick = np.where(ties.any(axis=-1), np.where(ties, idx, 99).min(axis=-1), idx.min(axis=-1))
    return np.sign(v) * E2M1[pick]


def _terms(xt, T, drop=0, flip=None, scale_err=None):
    """x_tilde as T e2m1 terms per 32-code group with 2^e from the group's
    maximum (the decode path's representation), with optional mistakes."""
    m, k = xt.shape
    out = np.zeros_like(xt)
    for g0 in range(0, k, 32):
        blk = xt[:, g0:g0 + 32]
        mx = np.abs(blk).max(axis=1, keepdims=True)
        e = np.frexp(mx)[1] - 2
        s = np.ldexp(1.0, e)
        if scale_err is not None and g0 == scale_err:
            s = 2 * s
        v = blk / np.ldexp(1.0, e)
        acc = np.zeros_like(v)
        for t in range(T - drop):
            q = _e2m1(v)
            assert np.all(np.abs(v) <= 4.0)
            acc += q * 8.0 ** -t
            v = (v - q) * 8.0
        if flip is not None and g0 == flip:
            acc = -acc
        out[:, g0:g0 + 32] = acc * s
    return out


@pytest.fixture(scope="module")
def layer():
    rng = np.random.default_rng(7)
    n, k, b, nb = 96, 2048, 128, 256
    keff = k // b * nb
    codes = W.random_codes(n, keff, O.TERNARY, 3)
    alpha = rng.random(n) * 0.05 + 0.01
    signs = np.where(rng.random(b) < 0.5, -1, 1).astype(np.int8)
    x = W.bf16_to_float(W.float_to_bf16(rng.standard_normal((2, k)).astype(np.float32)))
    yr = O.forward_code_domain(x, codes, alpha, b, nb, signs)
    xt = O.prep_activations(x, b, nb, signs)
    return x, codes, alpha, b, nb, signs, yr, xt


def test_e2m1_rounding_helper():
    v = np.array([0.2, 0.25, 0.3, 0.75, 1.25, 2.5, 3.4, 3.6, 5.0, -0.74])
    assert np.array_equal(_e2m1(v), [0.0, 0.0, 0.5, 1.0, 1.0, 2.0, 3.0, 4.0, 4.0, -0.5])


@pytest.mark.parametrize("T", [3, 4, 6])
def test_decode_arithmetic_within_bound(layer, T):
    x, codes, alpha, b, nb, signs, yr, xt = layer
    y = (_terms(xt, T) @ codes.T) * alpha
    EB.check(y, yr, EB.forward_bound(x, codes, alpha, b, nb, signs, T=T))


def test_prefill_arithmetic_within_bound(layer):
    x, codes, alpha, b, nb, signs, yr, xt = layer
    xb = W.bf16_to_float(W.float_to_bf16(xt.astype(np.float32))).astype(np.float64)
    y = (xb @ codes.T) * alpha
    EB.check(y, yr, EB.forward_bound(x, codes, alpha, b, nb, signs, T=None))


def test_one_term_too_few_fails(layer):
    x, codes, alpha, b, nb, signs, yr, xt = layer
    y = (_terms(xt, 3, drop=1) @ codes.T) * alpha
    with pytest.raises(AssertionError, match="rms"):
        EB.check(y, yr, EB.forward_bound(x, codes, alpha, b, nb, signs, T=3))


@pytest.mark.parametrize("mistake", ["flip", "scale"])
def test_one_group_wrong_fails(layer, mistake):
    x, codes, alpha, b, nb, signs, yr, xt = layer
    kw = {"flip": 2048} if mistake == "flip" else {"scale_err": 2048}
    y = (_terms(xt, 6, **kw) @ codes.T) * alpha
    with pytest.raises(AssertionError):
        EB.check(y, yr, EB.forward_bound(x, codes, alpha, b, nb, signs, T=6))


def test_transposed_batch_rows_fail(layer):
    x, codes, alpha, b, nb, signs, yr, xt = layer
    y = (_terms(xt[::-1].copy(), 6) @ codes.T) * alpha
    with pytest.raises(AssertionError):
        EB.check(y, yr, EB.forward_bound(x, codes, alpha, b, nb, signs, T=6))
