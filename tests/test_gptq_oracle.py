"""CPU pins of the oracle's GPTQ block compensation (Algorithm 1's update of
later columns), each checked against something other than the code itself:

* the factor: ``U`` upper triangular with ``U^T U H = I``;
* no calibration (``H = lambda I``, diagonal factor) or one block: the codes
  are those of the uncompensated encoder, bit for bit;
* every step's update equals the closed-form minimiser ``E H_FR H_RR^-1`` of
  the layer-output error over the later columns, computed from H by a linear
  solve (not from the factor); the normalised error solves ``E~ U_FF = E``;
* the method's purpose: the layer-output error ``tr(D H D^T)`` of the
  reconstructed weights falls against the uncompensated encoder;
* planted mistakes (the update without the normalisation, the factor
  transposed, a flipped sign) fail the closed-form check.
"""
import numpy as np
import pytest

import oracle as O
from paper_2510_03275_gb300 import workloads as W


def _layer(n=24, k=512, block=128, n_b=256, seed=5, tokens=None):
    rng = np.random.default_rng(seed)
    w = (rng.standard_normal((n, k)) * 0.02).astype(np.float32)
    x = W.calibration_activations(k, tokens or 2 * k, seed)
    h = O.gptq_hessian(x)
    u = O.gptq_factor(h)
    signs = np.where(rng.random(block) < 0.5, -1, 1).astype(np.int8)
    return w, h, u, block, n_b, signs


def test_factor_is_upper_cholesky_of_inverse():
    _, h, u, *_ = _layer()
    assert np.allclose(np.tril(u, -1), 0.0)
    assert np.all(np.diag(u) > 0)
    err = np.abs(u.T @ u @ h - np.eye(h.shape[0])).max()
    assert err < 1e-9, err


def test_hessian_definition():
    x = W.calibration_activations(64, 100, 3)
    h = O.gptq_hessian(x, damp_rel=0.0)
    # H_ij = 2 sum_t x_ti x_tj, element by element
    i, j = 5, 17
    assert np.isclose(h[i, j], 2.0 * sum(float(x[t, i]) * float(x[t, j]) for t in range(100)))
    hd = O.gptq_hessian(x, damp_rel=0.5)
    assert np.allclose(hd - h, 0.5 * np.mean(np.diag(h)) * np.eye(64))


@pytest.mark.parametrize("q", [O.TERNARY, O.BINARY])
def test_diagonal_factor_is_plain_encode(q):
    w, h, u, block, n_b, signs = _layer()
    ud = np.diag(np.full(w.shape[1], 3.0))          # H = I / 9: no cross terms
    c1, a1 = O.encode_gptq(w, ud, block, n_b, q, signs=signs)
    c0, a0 = O.encode(w, block, n_b, q, signs=signs)
    assert np.array_equal(c1, c0) and np.array_equal(a1, a0)


def test_single_block_is_plain_encode():
    w, h, u, block, n_b, signs = _layer(k=128)
    c1, a1 = O.encode_gptq(w, u, block, n_b, signs=signs)
    c0, a0 = O.encode(w, block, n_b, signs=signs)
    assert np.array_equal(c1, c0) and np.array_equal(a1, a0)


def _check_steps(steps, h, block, rtol=1e-4):
    """Each step's update W_after - W_before equals E H_FR H_RR^-1 with H
    restricted to the columns not yet quantized."""
    for b, st in enumerate(steps):
        f0 = b * block
        hs = h[f0:, f0:]
        hfr, hrr = hs[:block, block:], hs[block:, block:]
        want = st["E"].astype(np.float64) @ np.linalg.solve(hrr, hfr.T).T
        got = st["W_after"].astype(np.float64) - st["W_before"].astype(np.float64)
        scale = np.abs(want).max()
        assert scale > 0
        err = np.abs(got - want).max() / scale
        assert err < rtol, (b, err)


@pytest.mark.parametrize("q", [O.TERNARY, O.BINARY])
def test_update_is_the_closed_form_minimiser(q):
    w, h, u, block, n_b, signs = _layer()
    _, _, steps = O.encode_gptq(w, u, block, n_b, q, signs=signs, trace=True)
    assert len(steps) == w.shape[1] // block - 1
    _check_steps(steps, h, block)


def test_normalised_error_solves_triangular_system():
    w, h, u, block, n_b, signs = _layer()
    _, _, steps = O.encode_gptq(w, u, block, n_b, signs=signs, trace=True)
    u32 = u.astype(np.float32).astype(np.float64)
    for b, st in enumerate(steps):
        uff = u32[b * block:(b + 1) * block, b * block:(b + 1) * block]
        lhs = st["Et"].astype(np.float64) @ uff
        assert np.abs(lhs - st["E"]).max() <= 1e-5 * np.abs(st["E"]).max()


def test_error_is_weights_minus_reconstruction():
    """E of block 0 = W_F - alpha c G, with c the block's codes (reconstruct
    is the FFT definition of alpha Resample(c, B) Had^T)."""
    w, h, u, block, n_b, signs = _layer()
    codes, alpha, steps = O.encode_gptq(w, u, block, n_b, signs=signs, trace=True)
    rec = O.reconstruct(codes[:, :n_b], alpha, block, n_b, signs)
    assert np.abs(steps[0]["E"] - (w[:, :block] - rec)).max() < 1e-6


def test_compensation_lowers_layer_output_error():
    w, h, u, block, n_b, signs = _layer(n=32, k=768)
    cg, ag = O.encode_gptq(w, u, block, n_b, signs=signs)
    cp, ap = O.encode(w, block, n_b, signs=signs)
    w64 = w.astype(np.float64)

    def loss(c, a):
        d = w64 - O.reconstruct(c, a, block, n_b, signs)
        return float(np.einsum("ij,jk,ik->", d, h, d))

    lg, lp = loss(cg, ag), loss(cp, ap)
    assert lg < 0.85 * lp, (lg, lp)      # 0.75 on this seeded layer


@pytest.mark.parametrize("mistake", ["unnormalised", "transposed", "sign"])
def test_planted_update_mistakes_fail(mistake):
    w, h, u, block, n_b, signs = _layer()
    _, _, steps = O.encode_gptq(w, u, block, n_b, signs=signs, trace=True)
    u32 = u.astype(np.float32).astype(np.float64)
    bad = []
    for b, st in enumerate(steps):
        f0, f1 = b * block, (b + 1) * block
        e = st["E"].astype(np.float64)
        if mistake == "unnormalised":          # Algorithm 1's update taken literally
            upd = -(e @ u32[f0:f1, f1:])
        elif mistake == "transposed":          # the lower factor L = U^T in place of U
            lo = u32.T
            et = np.linalg.solve(lo[f0:f1, f0:f1].T, e.T).T
            upd = -(et @ lo[f0:f1, f1:])
        else:                                  # the update added instead of subtracted
            et = np.linalg.solve(u32[f0:f1, f0:f1].T, e.T).T
            upd = et @ u32[f0:f1, f1:]
        wb = st["W_before"].astype(np.float64)
        bad.append(dict(st, W_after=wb + upd))
    with pytest.raises(AssertionError):
        _check_steps(bad, h, block)
