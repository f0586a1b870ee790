"""CPU: the error bounds the GPU parity tests apply (tests/errbound.py)
against an fp64 emulation of each path's arithmetic (decode terms, the bf16
prefill operand, the dense route's bf16 rebuilt weights), and against
planted mistakes in that emulation: the bounds must hold for the arithmetic
as described and fail for a term too few, a flipped sign, a wrong scale,
coarser weights, a wrong G or misplaced blocks."""
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


def _dense_y(x, codes, alpha, b, nb, signs, mant_bits=8, g=None, shift=0):
    """The dense route's arithmetic in fp64: W'' = 2 C G per block, rounded
    to `mant_bits` significant bits (8: bf16), y = alpha / 2 x W''^T; with
    optional mistakes (another G, blocks of codes shifted by `shift`)."""
    g = O.decode_table(b, nb, signs, True) if g is None else g
    c = np.asarray(codes, dtype=np.float64)
    rows, keff = c.shape
    nblk = keff // nb
    cb = np.roll(c.reshape(rows, nblk, nb), shift, axis=1)
    w2 = 2.0 * (cb @ g).reshape(rows, nblk * b)
    e = np.floor(np.log2(np.maximum(np.abs(w2), 1e-300)))
    q = 2.0 ** (e - (mant_bits - 1))
    w2r = np.where(w2 == 0, 0.0, np.round(w2 / q) * q)
    return (np.asarray(x, dtype=np.float64) @ w2r.T) * (alpha / 2.0)


def test_dense_arithmetic_within_bound(layer):
    x, codes, alpha, b, nb, signs, yr, xt = layer
    y = _dense_y(x, codes, alpha, b, nb, signs)
    EB.check(y, yr, EB.forward_bound(x, codes, alpha, b, nb, signs, dense=True))


def test_dense_rebuilt_weights_are_c_times_g(layer):
    """W' = C G reproduces the code-domain forward exactly (associativity):
    x W'^T = C x_tilde per row, in fp64."""
    x, codes, alpha, b, nb, signs, yr, xt = layer
    wp = EB.rebuilt_weights(codes, b, nb, signs)
    np.testing.assert_allclose((x @ wp.T) * alpha, yr, rtol=1e-10, atol=1e-12 * np.abs(yr).max())


@pytest.mark.parametrize("mistake", ["coarse", "signs", "shift"])
def test_dense_mistakes_fail(layer, mistake):
    x, codes, alpha, b, nb, signs, yr, xt = layer
    if mistake == "coarse":      # weights rounded to 4 significant bits instead of 8
        y = _dense_y(x, codes, alpha, b, nb, signs, mant_bits=4)
    elif mistake == "signs":     # G built without the Hadamard signs
        y = _dense_y(x, codes, alpha, b, nb, signs, g=O.decode_table(b, nb, np.ones_like(signs), True))
    else:                        # each block's weights rebuilt from the next block's codes
        y = _dense_y(x, codes, alpha, b, nb, signs, shift=1)
    with pytest.raises(AssertionError):
        EB.check(y, yr, EB.forward_bound(x, codes, alpha, b, nb, signs, dense=True))
