"""Per-element error bounds of the CUDA forward against the oracle's fp64
result, derived from the arithmetic each path performs (test
infrastructure: the bounds use the oracle's x_tilde and G, nothing of the
CUDA path).

Both paths compute y[m, r] = alpha_r * sum_j c[r, j] x_tilde[m, j]
(section 3.5, eq. 12) with x_tilde = G x per input block, and differ from the
fp64 oracle by

  decode (M <= 64)   x_tilde carried as T e2m1 terms per batch row and
                     32-code group g of a 128-code block:
                     x_tilde ~ 2^e sum_t 8^-t q_t with 2^e <= max_g |x_tilde| / 2
                     and |x_tilde 2^-e| < 4.  Round-to-nearest onto the e2m1
                     grid leaves at most 0.5 (the grid spacing in [2, 4) is
                     1; residuals are scaled by 8 and stay within 4), so after
                     T terms |error| <= 0.5 * 8^-(T-1) * 2^e
                                   <= 0.25 * 8^-(T-1) * max_g |x_tilde|.
                     The group maximum is bounded by the 128-code block's.
  prefill (M > 64)   x_tilde rounded once to bf16 (8 significant bits):
                     |error| <= 2^-8 |x_tilde_j|.
  dense (large M)    the route that rebuilds the weights: W'' = 2 C G per
                     block in fp32 (G as bf16 hi + lo, ~2^-16), rounded once
                     to bf16 (|delta W''_rk| <= 2^-9 |W''_rk|), then
                     y = alpha / 2 x W''^T.  Since |W''_rk| <= 2 sum_j |c_rj|
                     |G_jk|, the error is at most alpha (2^-9 + 2^-16)
                     sum_j |c_rj| sum_k |G_jk| |x_k|: a per-code term of
                     2^-9 sum_i |G_ji x_i| in the sum below.

plus, for both, the fp32 work: x_tilde from bf16 x and G split into two
bf16 parts (about 2^-16 of sum_i |G_ji x_i|), and fp32 accumulation over K
and the split-K partials.  That part is covered by 2^-12 * sum_j |c_rj|
sum_i |G_ji| |x_i|, generous for K up to 2^16 codes and still far below the
error of a dropped term, a wrong scale, sign or index.

The worst-case bound grows with K where independent rounding errors grow
with sqrt(K), so ``check`` also bounds the root-mean-square error by twice
what independent errors, each uniform within its bound, would give: one term
fewer than the path's T, or a rounding that ignores the lower terms, is then
several times over.
"""
import numpy as np

import oracle as O

FP32_SLACK = 2.0 ** -12


def _gx_abs(x, block, n_b, signs, hadamard):
    """sum_i |G_ji| |x_i| per batch row and code j (fp64)."""
    g = np.abs(O.decode_table(block, n_b, signs, hadamard))
    x = np.abs(np.asarray(x, dtype=np.float64))
    m, k = x.shape
    return (x.reshape(m, k // block, block) @ g.T).reshape(m, -1)


class Bound(np.ndarray):
    """Per-element bound with the expected root-mean-square error attached
    (``rms``)."""


def forward_bound(x, codes, alpha, block, n_b, signs, T=None, hadamard=True, dense=False):
    """Per-element bound on |y_cuda - y_oracle| for batch rows x (M, K) and
    the output rows whose codes are ``codes`` (rows, K_eff) and scales
    ``alpha``.  T: e2m1 terms of the decode path; None for the bf16 prefill
    path; dense: the route that rebuilds the weights in bf16."""
    if dense:
        return _dense_bound(x, codes, alpha, block, n_b, signs, hadamard)
    xt = O.prep_activations(x, block, n_b, signs, hadamard)
    m, keff = xt.shape
    if T is None:
        per = 2.0 ** -8 * np.abs(xt)
    else:
        nblk = (keff + 127) // 128
        pad = np.zeros((m, nblk * 128))
        pad[:, :keff] = np.abs(xt)
        mx = pad.reshape(m, nblk, 128).max(axis=2)
        per = np.repeat(0.25 * 8.0 ** -(T - 1) * mx, 128, axis=1)[:, :keff] * (1 + 1e-6)
    slack = FP32_SLACK * _gx_abs(x, block, n_b, signs, hadamard)
    c = np.abs(np.asarray(codes, dtype=np.float64))
    a = np.abs(np.asarray(alpha, dtype=np.float64))[None, :]
    b = ((per + slack) @ c.T) * a + 1e-30
    # independent errors uniform within +-per: variance per^2 / 3 each
    var = ((per ** 2 / 3.0) @ (c ** 2).T) * a ** 2
    out = np.asarray(b).view(Bound)
    # the fp32 part, as independent errors of at most `slack` per code
    var = var + ((slack ** 2) @ (c ** 2).T) * a ** 2
    out.rms = float(np.sqrt(var.mean())) + 1e-30
    return out


def rebuilt_weights(codes, block, n_b, signs, hadamard=True):
    """W' = C G per block (fp64): the weights the dense route rebuilds (up
    to its factor 2 and the bf16 rounding), rows x K."""
    g = O.decode_table(block, n_b, signs, hadamard)           # n_b x B
    c = np.asarray(codes, dtype=np.float64)
    rows, keff = c.shape
    nblk = keff // n_b
    return (c.reshape(rows, nblk, n_b) @ g).reshape(rows, nblk * block)


def _dense_bound(x, codes, alpha, block, n_b, signs, hadamard):
    gx = _gx_abs(x, block, n_b, signs, hadamard)              # M x K_eff
    c = np.abs(np.asarray(codes, dtype=np.float64))
    a = np.abs(np.asarray(alpha, dtype=np.float64))[None, :]
    per = (2.0 ** -9 + 2.0 ** -16) * gx
    slack = FP32_SLACK * gx
    b = ((per + slack) @ c.T) * a + 1e-30
    out = np.asarray(b).view(Bound)
    # independent roundings of the rebuilt weights, each uniform within
    # +-2^-9 |W''_rk| = +-2^-8 |W'_rk|: error_r = alpha / 2 sum_k x_k dW''_rk
    wp = rebuilt_weights(codes, block, n_b, signs, hadamard)
    xf = np.asarray(x, dtype=np.float64)
    var = ((xf ** 2) @ (wp ** 2).T) * (2.0 ** -18 / 3.0) * a ** 2
    var = var + ((slack ** 2) @ (c ** 2).T) * a ** 2
    out.rms = float(np.sqrt(var.mean())) + 1e-30
    return out


def elementwise_error(y, yr):
    """max |y - y_ref| / max(|y_ref|, 1e-3 max |y_ref|) over all elements."""
    y = np.asarray(y, dtype=np.float64)
    yr = np.asarray(yr, dtype=np.float64)
    floor = 1e-3 * np.abs(yr).max()
    return float((np.abs(y - yr) / np.maximum(np.abs(yr), floor)).max())


def check(y, yr, bound, what=""):
    """Assert every element within its bound and the root-mean-square error
    within twice the expected one; return the element-wise error."""
    y = np.asarray(y, dtype=np.float64)
    d = np.abs(y - yr)
    bound = np.asarray(bound) if not isinstance(bound, Bound) else bound
    bad = d > np.asarray(bound)
    elem = elementwise_error(y, yr)
    rms = float(np.sqrt((d ** 2).mean()))
    if hasattr(bound, "rms") and rms > 2.0 * bound.rms:
        raise AssertionError(f"{what}: rms error {rms:.3e} over twice the expected {bound.rms:.3e}; "
                             f"element-wise error {elem:.3e}")
    if bad.any():
        i = np.unravel_index(np.argmax(d / bound), d.shape)
        raise AssertionError(f"{what}: {int(bad.sum())} of {d.size} elements beyond the bound; worst "
                             f"{tuple(int(v) for v in i)}: |d|={d[i]:.3e} bound={bound[i]:.3e} "
                             f"ref={yr[i]:.3e}; element-wise error {elem:.3e}")
    return elem
