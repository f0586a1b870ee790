"""SDQ-LLM oracle: plain, slow, obviously-correct CPU definitions (numpy).

TEST INFRASTRUCTURE ONLY -- see ``oracle/__init__.py``.  Product code must
never import this module.

What it computes (SDQ-LLM, arXiv 2510.03275):

* Sylvester Hadamard matrix, eq. (13); the "random Hadamard matrix" of
  Algorithm 1 read as ``Had = diag(d) . H_B / sqrt(B)`` with a sign vector
  ``d`` that is passed in (it is an input of the method, drawn by the seeded
  input generator).
* The Resample function of Algorithm 1 (FFT, zero-pad or truncate, the
  Nyquist-bin rule, inverse FFT, gain ``N_new/d_col``).
* SDQuant of Algorithm 1 with the first-order Sigma-Delta recursion of
  eqs. (7)-(8) and the quantizers of eqs. (3)-(6).
* The per-row scale alpha (section 3.1: "alpha ... typically mean(|W|)").
* Reconstruction ``W_hat_blk = alpha * Resample(codes, B) . Had^T``
  (Algorithm 1, outer loop) and the dense reference forward ``x . W_hat^T``.
* The code-domain forward ``y = alpha * C . (G x)``, ``G = D^T Had^T``: the
  exact adjoint of the decimation, which is how activations are "upsampled
  with the same OSR" at inference (section 3.5, Fig. 5, with eq. (12)).
* Storage accounting, eq. (14).
* The packed code layouts (plain and tiled) of the C-ABI header, and the
  base-3 storage of ternary codes (5 trits per byte, 1.6 bits per code).

Readings of points the paper leaves open:

* Integrator: eq. (8) ``i_n = i_{n-1} + x_n - y_{n-1}`` (accumulating form);
  Algorithm 1's SDQuant body writes the integrator without the accumulation,
  which contradicts eq. (8) and the Z-domain analysis of eqs. (9)-(11).
* fp32 order of eq. (8): ``(i + x) - y_prev``, left to right, no FMA.
* Integrator and previous output reset to 0 at the start of every block of B
  columns (SDQuant is called per block and initialises both to zero).
* alpha: per output row.  Default ``max |x_up|`` over the upsampled row
  (``ALPHA_MAXABS``); ``mean |x_up|`` (``ALPHA_MEANABS``) kept as an option.
* Ternary threshold ``theta = 0.5 * alpha`` with ``|i| == theta -> 0``
  (eq. (6) is closed at +-theta); binary ``sign(0) = +1`` (eq. (4)).
* Resample Nyquist rule applied at bin ``m/2`` with ``m = min(N_new, d_col)``
  and only when ``m`` is even: upsampling splits the bin half-and-half into
  bins ``m/2`` and ``N_new - m/2``; downsampling folds ``X[m/2] + X[d-m/2]``.
  The inverse FFT carries numpy's ``1/N_new`` factor, then the gain
  ``N_new/d_col`` of Algorithm 1 is applied, so amplitudes are preserved.
* OSR is rational, ``OSR = n_b / B`` with ``n_b`` an integer.
* GPTQ block compensation (Algorithm 1's update of later columns with the
  inverse Hessian): :func:`encode` leaves it out (with no calibration data
  the Hessian is ``lambda I`` and the update vanishes, so blocks are
  independent); :func:`encode_gptq` applies it with a given factor of
  ``H^-1``, reading the update as the exact block update ``E U_FF^-1 U_FR``
  (Algorithm 1 prints ``E . H^-1_{F,R}``), with alpha from the original
  weights.

Canonical fp32 mode (the bit-exact contract with the CUDA encoder): the
composed table ``A_enc = fp32(U . Had^T)`` is built in fp64 and rounded once;
``x_up[j] = fl(...fl(fl(A[j,0] w_0) + fl(A[j,1] w_1)) ... )`` with every
product and sum rounded to fp32 in ascending ``k`` (numpy elementwise float32
ops never fuse a multiply-add); the scan runs in fp32 in the order above.
"""
from __future__ import annotations

import math

import numpy as np

# Quantizer ids: the value is the number of storage bits per code.
BINARY = 1
TERNARY = 2
# |entry| below this in the fp64 encode table is fp64 noise on an exact zero.
ZERO_FLUSH = 2.0 ** -46
# alpha modes.
ALPHA_MAXABS = 0
ALPHA_MEANABS = 1

__all__ = [
    "BINARY", "TERNARY", "ALPHA_MAXABS", "ALPHA_MEANABS",
    "sylvester_hadamard", "hadamard_matrix", "resample", "resample_matrix",
    "encode_table", "decode_table", "upsample_canonical", "row_alpha",
    "sigma_delta_scan", "sigma_delta_scan_f64", "encode", "encode_f64",
    "reconstruct", "forward", "forward_code_domain", "prep_activations",
    "compression_ratio", "plain_words_per_row", "pack_plain", "unpack_plain",
    "tiled_geometry", "pack_tiled", "unpack_tiled",
    "gptq_hessian", "gptq_factor", "decode_table32", "encode_gptq",
    "TRITS_PER_BYTE", "base3_bytes_per_row", "pack_base3", "unpack_base3",
]


# --------------------------------------------------------------------------
# Hadamard (section 3.3, eq. (13))
# --------------------------------------------------------------------------
def sylvester_hadamard(n: int) -> np.ndarray:
    """Sylvester construction of eq. (13): H_1 = [1], H_2k = [[H, H], [H, -H]].

    Returns an int64 matrix with ``H @ H.T == n I``.  ``n`` must be a power
    of two.
    """
    if n < 1 or n & (n - 1):
        raise ValueError("Sylvester Hadamard size must be a power of two")
    h = np.ones((1, 1), dtype=np.int64)
    while h.shape[0] < n:
        h = np.block([[h, h], [h, -h]])
    return h


def hadamard_matrix(block: int, signs=None, enabled: bool = True) -> np.ndarray:
    """The "random Hadamard matrix" Had of Algorithm 1 (fp64, B x B).

    Read as ``diag(d) . H_B / sqrt(B)``: orthonormal (Algorithm 1 inverts it
    with ``Had^T``), randomised by the sign vector ``d`` (+-1, length B) on the
    input side.  ``signs=None`` means all +1.  ``enabled=False`` gives the
    identity (the "Hadamard N" rows of the Table 2 ablation).
    """
    if not enabled:
        return np.eye(block)
    d = np.ones(block) if signs is None else np.asarray(signs, dtype=np.float64)
    if d.shape != (block,) or not np.all(np.abs(d) == 1):
        raise ValueError("signs must be a length-B vector of +-1")
    return d[:, None] * sylvester_hadamard(block).astype(np.float64) / math.sqrt(block)


# --------------------------------------------------------------------------
# Resample (Algorithm 1, function Resample)
# --------------------------------------------------------------------------
def resample(w, n_new: int) -> np.ndarray:
    """Band-limited FFT resampling of each row of ``w`` to ``n_new`` samples.

    Steps in the order of Algorithm 1's Resample: FFT of the row; keep the
    ``m = min(n_new, d_col)`` lowest frequencies (zero-pad or truncate); apply
    the Nyquist-bin rule when ``m`` is even (halve and mirror on upsample,
    fold the two aliases on downsample); inverse FFT (numpy's ``1/n_new``);
    take the real part; multiply by ``n_new / d_col``.
    """
    w = np.atleast_2d(np.asarray(w, dtype=np.float64))
    d = w.shape[1]
    X = np.fft.fft(w, axis=1)
    m = min(n_new, d)
    h = (m - 1) // 2              # strictly positive bins kept on each side
    Y = np.zeros((w.shape[0], n_new), dtype=np.complex128)
    Y[:, 0] = X[:, 0]
    if h > 0:
        Y[:, 1:h + 1] = X[:, 1:h + 1]
        Y[:, n_new - h:] = X[:, d - h:]
    if m % 2 == 0 and m >= 2:
        ny = m // 2
        if n_new > d:             # upsample: split the Nyquist bin
            Y[:, ny] = 0.5 * X[:, ny]
            Y[:, n_new - ny] = 0.5 * X[:, ny]
        elif n_new < d:           # downsample: fold both aliases into bin m/2
            Y[:, ny] = X[:, ny] + X[:, d - ny]
        else:                     # same length: identity
            Y[:, ny] = X[:, ny]
    y = np.fft.ifft(Y, axis=1)
    return np.real(y) * (n_new / d)


def resample_matrix(d: int, n_new: int) -> np.ndarray:
    """R (d x n_new) with ``resample(v, n_new) == v @ R`` for a row ``v``."""
    return resample(np.eye(d), n_new)


def _check_geometry(block: int, n_b: int):
    if block < 1 or block & (block - 1):
        raise ValueError("block size B must be a power of two")
    if n_b < block:
        raise ValueError("OSR must be >= 1 (n_b >= B)")


def encode_table(block: int, n_b: int, signs=None, hadamard: bool = True) -> np.ndarray:
    """Canonical encode table ``A_enc = fp32(U . Had^T)`` (n_b x B).

    For one row block ``w`` (length B), Algorithm 1 forms ``v = w . Had`` and
    ``x_up = Resample(v, n_b)``; by linearity ``x_up = A_enc w`` with
    ``A_enc = (Had . R)^T``.  Built in fp64 and rounded to fp32 once.
    """
    _check_geometry(block, n_b)
    had = hadamard_matrix(block, signs, hadamard)
    a64 = (had @ resample_matrix(block, n_b)).T
    # Entries that are exactly zero in real arithmetic (e.g. the interpolating
    # property of Resample at integer OSR, and cancellations of the Hadamard
    # rows) come out of fp64 as +-1e-16 noise; they are set to exact zero so
    # that the fp32 table does not depend on how the fp64 value was computed.
    a64[np.abs(a64) < ZERO_FLUSH] = 0.0
    return a64.astype(np.float32)


def decode_table(block: int, n_b: int, signs=None, hadamard: bool = True) -> np.ndarray:
    """Activation transform ``G = D^T . Had^T`` (n_b x B, fp64).

    The reconstructed block is ``w_hat = alpha * Resample(c, B) . Had^T =
    alpha * (c . D) . Had^T`` with ``D = resample_matrix(n_b, B)``, so
    ``w_hat . x_b = alpha * c . (D Had^T x_b) = alpha * c . (G x_b)``.
    """
    _check_geometry(block, n_b)
    had = hadamard_matrix(block, signs, hadamard)
    return resample_matrix(n_b, block) @ had.T


# --------------------------------------------------------------------------
# Canonical fp32 encoder (Algorithm 1 without compensation, eqs. (3)-(8))
# --------------------------------------------------------------------------
def _blocks(W, block: int) -> np.ndarray:
    W = np.asarray(W)
    n, k = W.shape
    if k % block:
        raise ValueError("d_col must be a multiple of the block size B")
    return W.reshape(n, k // block, block)


def upsample_canonical(W, a_enc32: np.ndarray) -> np.ndarray:
    """x_up (N, K/B, n_b) fp32 in the canonical operation order.

    ``x_up[r, b, j] = fl(... fl(fl(A[j,0] w_0) + fl(A[j,1] w_1)) ...)`` with
    ``w = W[r, bB:(b+1)B]``: each product and each partial sum rounded to
    fp32, ``k`` ascending.  Loops over ``k`` with float32 elementwise ops.
    """
    a = np.asarray(a_enc32, dtype=np.float32)
    n_b, block = a.shape
    wb = _blocks(np.asarray(W, dtype=np.float32), block)
    x = wb[:, :, 0:1] * a[None, None, :, 0]
    for k in range(1, block):
        x = x + wb[:, :, k:k + 1] * a[None, None, :, k]
    assert x.dtype == np.float32
    return x


def row_alpha(x_up: np.ndarray, mode: int = ALPHA_MAXABS) -> np.ndarray:
    """Per-row scale alpha (section 3.1) over the whole upsampled row, fp32.

    MAXABS: ``max |x_up|`` (exact in any order).  MEANABS: fp32 sum of
    ``|x_up|`` taken sequentially in (block, index) order, divided (IEEE fp32)
    by the upsampled row length.
    """
    n = x_up.shape[0]
    flat = np.abs(x_up.reshape(n, -1)).astype(np.float32)
    if mode == ALPHA_MAXABS:
        return flat.max(axis=1).astype(np.float32)
    if mode == ALPHA_MEANABS:
        s = np.add.accumulate(flat, axis=1, dtype=np.float32)[:, -1]
        return (s / np.float32(flat.shape[1])).astype(np.float32)
    raise ValueError("unknown alpha mode")


def sigma_delta_scan(x: np.ndarray, alpha: np.ndarray, quantizer: int,
                     return_state: bool = False):
    """First-order Sigma-Delta scan of eqs. (7)-(8) in fp32, per block.

    ``x``: (N, nblk, n_b) fp32; ``alpha``: (N,) fp32.  For every (row, block)
    the integrator ``i`` and previous output start at 0 (SDQuant), then for
    each sample ``i = fl(fl(i + x_n) - y_prev)``, ``q = Q(i)`` and
    ``y_prev = q * alpha``.  Ternary Q is eq. (6) with ``theta = alpha/2``;
    binary Q is eq. (4).  Returns int8 codes (N, nblk, n_b); with
    ``return_state`` also the integrator values (same shape, fp32).
    """
    x = np.asarray(x, dtype=np.float32)
    a = np.asarray(alpha, dtype=np.float32)[:, None]
    theta = (a * np.float32(0.5)).astype(np.float32)
    i = np.zeros(x.shape[:2], dtype=np.float32)
    yp = np.zeros(x.shape[:2], dtype=np.float32)
    codes = np.zeros(x.shape, dtype=np.int8)
    states = np.zeros(x.shape, dtype=np.float32) if return_state else None
    for n in range(x.shape[2]):
        i = (i + x[:, :, n]) - yp
        if quantizer == TERNARY:
            q = np.where(i > theta, 1, np.where(i < -theta, -1, 0)).astype(np.int8)
        elif quantizer == BINARY:
            q = np.where(i >= 0, 1, -1).astype(np.int8)
        else:
            raise ValueError("unknown quantizer")
        codes[:, :, n] = q
        yp = (q.astype(np.float32) * a).astype(np.float32)
        if return_state:
            states[:, :, n] = i
    return (codes, states) if return_state else codes


def encode(W, block: int, n_b: int, quantizer: int = TERNARY,
           alpha_mode: int = ALPHA_MAXABS, signs=None, hadamard: bool = True):
    """Canonical fp32 SDQ encoder (Algorithm 1, SDQuant, eqs. (3)-(8)).

    Returns ``(codes, alpha)``: int8 codes (N, K/B * n_b) in {-1,0,1}
    (ternary) or {-1,1} (binary), block b occupying columns
    ``[b*n_b, (b+1)*n_b)`` as in Algorithm 1's ``Q_out``; alpha fp32 (N,).
    """
    a32 = encode_table(block, n_b, signs, hadamard)
    x = upsample_canonical(W, a32)
    alpha = row_alpha(x, alpha_mode)
    codes = sigma_delta_scan(x, alpha, quantizer)
    return codes.reshape(codes.shape[0], -1), alpha


# --------------------------------------------------------------------------
# fp64 reference mode (real-arithmetic reading, for the theory pins)
# --------------------------------------------------------------------------
def sigma_delta_scan_f64(x, alpha, quantizer: int):
    """Eqs. (7)-(8) in fp64 on a (..., n) array with per-leading-index alpha.

    Returns ``(codes, i, y)``: codes in {-1,0,1}, the integrator i_n and the
    outputs y_n = alpha * q_n, all with the shape of ``x``.
    """
    x = np.asarray(x, dtype=np.float64)
    a = np.asarray(alpha, dtype=np.float64)
    if a.ndim == x.ndim:          # alpha given with a trailing unit axis
        a = a[..., 0]
    a = np.broadcast_to(a, x.shape[:-1])
    i = np.zeros(x.shape[:-1])
    yp = np.zeros(x.shape[:-1])
    codes = np.zeros(x.shape, dtype=np.int8)
    ii = np.zeros(x.shape)
    yy = np.zeros(x.shape)
    for n in range(x.shape[-1]):
        i = i + x[..., n] - yp
        if quantizer == TERNARY:
            q = np.where(i > a / 2, 1, np.where(i < -a / 2, -1, 0))
        else:
            q = np.where(i >= 0, 1, -1)
        codes[..., n] = q
        yp = q * a
        ii[..., n] = i
        yy[..., n] = yp
    return codes, ii, yy


def encode_f64(W, block: int, n_b: int, quantizer: int = TERNARY,
               alpha_mode: int = ALPHA_MAXABS, signs=None, hadamard: bool = True):
    """Algorithm 1 in fp64 via the FFT Resample (no canonical rounding)."""
    W = np.asarray(W, dtype=np.float64)
    had = hadamard_matrix(block, signs, hadamard)
    wb = _blocks(W, block)
    n, nblk, _ = wb.shape
    v = wb @ had                                    # w . Had per block
    x = resample(v.reshape(n * nblk, block), n_b).reshape(n, nblk, n_b)
    flat = np.abs(x.reshape(n, -1))
    alpha = flat.max(axis=1) if alpha_mode == ALPHA_MAXABS else flat.mean(axis=1)
    codes, _, _ = sigma_delta_scan_f64(x, alpha[:, None], quantizer)
    return codes.reshape(n, -1), alpha


# --------------------------------------------------------------------------
# Reconstruction and forward (Algorithm 1 outer loop; section 3.5; eq. (12))
# --------------------------------------------------------------------------
def reconstruct(codes, alpha, block: int, n_b: int, signs=None,
                hadamard: bool = True) -> np.ndarray:
    """W_hat (N, K) fp64: per block ``alpha_r * Resample(c_rb, B) . Had^T``."""
    codes = np.asarray(codes, dtype=np.float64)
    n = codes.shape[0]
    nblk = codes.shape[1] // n_b
    had = hadamard_matrix(block, signs, hadamard)
    c = codes.reshape(n * nblk, n_b)
    wb = resample(c, block) @ had.T
    return np.asarray(alpha, dtype=np.float64)[:, None] * wb.reshape(n, nblk * block)


def forward(x, w_hat) -> np.ndarray:
    """Dense reference forward ``y = x . W_hat^T`` in fp64 (x: (M, K))."""
    return np.asarray(x, dtype=np.float64) @ np.asarray(w_hat, dtype=np.float64).T


def prep_activations(x, block: int, n_b: int, signs=None, hadamard: bool = True):
    """x_tilde (M, K/B * n_b) fp64: ``G x_b`` for every block b of x."""
    x = np.asarray(x, dtype=np.float64)
    m, k = x.shape
    g = decode_table(block, n_b, signs, hadamard)
    xb = x.reshape(m, k // block, block)
    return (xb @ g.T).reshape(m, -1)


def forward_code_domain(x, codes, alpha, block: int, n_b: int, signs=None,
                        hadamard: bool = True, rows=None) -> np.ndarray:
    """``y[m, r] = alpha_r * sum_j c[r, j] * x_tilde[m, j]`` in fp64.

    Equal to ``forward(x, reconstruct(...))`` by construction of G; with
    ``rows`` only those output rows are computed (for sampled checks).
    """
    xt = prep_activations(x, block, n_b, signs, hadamard)
    c = np.asarray(codes)
    a = np.asarray(alpha, dtype=np.float64)
    if rows is not None:
        c = c[rows]
        a = a[rows]
    return (xt @ c.astype(np.float64).T) * a[None, :]


# --------------------------------------------------------------------------
# Storage accounting (eq. (14))
# --------------------------------------------------------------------------
def compression_ratio(bits_per_code: float, osr: float) -> float:
    """Eq. (14): eta = N * OSR / 16 (N = bits per code; 1.58 for ternary)."""
    return bits_per_code * osr / 16.0


# --------------------------------------------------------------------------
# Packed layouts (defined in include/sdq.h)
# --------------------------------------------------------------------------
def _field(code: int, quantizer: int) -> int:
    if quantizer == TERNARY:
        return {0: 0, 1: 1, -1: 3}[int(code)]
    return 1 if code > 0 else 0


def plain_words_per_row(k_eff: int, quantizer: int) -> int:
    """uint32 words per row of the plain layout: rows padded to 128 bits."""
    bits = k_eff * quantizer
    return ((bits + 127) // 128) * 4


def pack_plain(codes, quantizer: int) -> np.ndarray:
    """Plain layout: code j of row r sits in uint32 word ``r*W + j // (32/b)``
    at bit ``b * (j mod (32/b))`` (b = bits per code).  Ternary fields:
    00 = 0, 01 = +1, 11 = -1.  Binary: 1 = +1, 0 = -1.  Padding fields 0."""
    codes = np.asarray(codes)
    n, k = codes.shape
    b = quantizer
    per = 32 // b
    wpr = plain_words_per_row(k, quantizer)
    out = np.zeros((n, wpr), dtype=np.uint64)
    if quantizer == TERNARY:
        fld = np.where(codes == 1, 1, np.where(codes == -1, 3, 0)).astype(np.uint64)
        if np.any((codes != 0) & (codes != 1) & (codes != -1)):
            raise ValueError("ternary codes must be in {-1,0,1}")
    else:
        if np.any((codes != 1) & (codes != -1)):
            raise ValueError("binary codes must be in {-1,1}")
        fld = (codes > 0).astype(np.uint64)
    j = np.arange(k)
    for jj in range(per):
        sel = j[jj::per]
        out[:, sel // per] |= fld[:, sel] << np.uint64(b * jj)
    return out.astype(np.uint32)


def unpack_plain(words, quantizer: int, k_eff: int) -> np.ndarray:
    """Inverse of :func:`pack_plain` (ternary pattern 10 decodes to 0)."""
    words = np.asarray(words, dtype=np.uint64)
    b = quantizer
    per = 32 // b
    j = np.arange(k_eff)
    f = (words[:, j // per] >> (np.uint64(b) * (j % per).astype(np.uint64))) & np.uint64((1 << b) - 1)
    if quantizer == TERNARY:
        return np.where(f == 1, 1, np.where(f == 3, -1, 0)).astype(np.int8)
    return np.where(f == 1, 1, -1).astype(np.int8)


TILE_ROWS = 128      # rows per tile of the tiled layout
GROUP_CODES = 64     # codes per k group of the tiled layout


def tiled_geometry(n_out: int, k_eff: int, quantizer: int):
    """(tiles, k groups per tile, words per row per group) of the tiled
    layout.  K_eff is padded to a multiple of 128 codes."""
    k_pad = -(-k_eff // 128) * 128
    wpr = GROUP_CODES * quantizer // 32
    return -(-n_out // TILE_ROWS), k_pad // GROUP_CODES, wpr


def _tiled_position(row: int, k: int, quantizer: int, n_groups: int):
    """(word index, bit shift) of code (row, k) in the tiled layout.

    Rows are cut into tiles of 128 (T = row // 128, r = row % 128) and codes
    into groups of 64 (G = k // 64).  Slab (T, G) is 128 * wpr consecutive
    uint32 words starting at word ``128 * wpr * (T * n_groups + G)``, and row
    r owns the ``wpr`` words starting at ``wpr * r`` inside it (wpr = 4
    ternary, 2 binary).  Inside the row's words the codes keep their natural
    order: ternary word i = (k % 64) // 16 holds k at field f = k % 16 (bits
    2f, 2f+1); binary word i = (k % 64) // 32 holds k at bit f = k % 32.
    """
    T, r = divmod(row, TILE_ROWS)
    G, kk = divmod(k, GROUP_CODES)
    wpr = GROUP_CODES * quantizer // 32
    per = 32 // quantizer
    i, f = divmod(kk, per)
    word = wpr * (TILE_ROWS * (T * n_groups + G) + r) + i
    return word, quantizer * f


def pack_tiled(codes, quantizer: int) -> np.ndarray:
    """Tiled layout (see :func:`_tiled_position`), padding fields 0.

    Pure-Python loop over every code: use on small matrices only.
    """
    codes = np.asarray(codes)
    n, k = codes.shape
    nt, ng, wpr = tiled_geometry(n, k, quantizer)
    out = [0] * (nt * ng * TILE_ROWS * wpr)
    for r in range(n):
        for kk in range(k):
            fv = _field(codes[r, kk], quantizer)
            if fv:
                w, s = _tiled_position(r, kk, quantizer, ng)
                out[w] |= fv << s
    return np.array(out, dtype=np.uint64).astype(np.uint32)


def unpack_tiled(words, quantizer: int, n_out: int, k_eff: int) -> np.ndarray:
    """Inverse of :func:`pack_tiled` (pure-Python loop; small matrices)."""
    words = [int(v) for v in np.asarray(words, dtype=np.uint32)]
    _, ng, _ = tiled_geometry(n_out, k_eff, quantizer)
    out = np.zeros((n_out, k_eff), dtype=np.int8)
    mask = (1 << quantizer) - 1
    for r in range(n_out):
        for kk in range(k_eff):
            w, s = _tiled_position(r, kk, quantizer, ng)
            f = (words[w] >> s) & mask
            if quantizer == TERNARY:
                out[r, kk] = 1 if f == 1 else (-1 if f == 3 else 0)
            else:
                out[r, kk] = 1 if f else -1
    return out


# --------------------------------------------------------------------------
# Base-3 storage of ternary codes (eq. (14)'s ~1.58 bits: 5 trits per byte)
# --------------------------------------------------------------------------
TRITS_PER_BYTE = 5


def base3_bytes_per_row(k_eff: int) -> int:
    """Bytes per row of the base-3 layout: ceil(K_eff / 5) rounded up to a
    multiple of 16."""
    return 16 * ((-(-k_eff // TRITS_PER_BYTE) + 15) // 16)


def pack_base3(codes) -> np.ndarray:
    """Ternary codes (N, K_eff) -> base-3 bytes (N, bytes_per_row) uint8.

    Code j of a row is trit ``t = code mod 3`` (0 -> 0, +1 -> 1, -1 -> 2) at
    digit ``j mod 5`` of byte ``j // 5``: ``byte = sum_d t_d 3^d``, at most
    242.  Codes past K_eff and padding bytes are 0.
    """
    c = np.asarray(codes)
    n, k = c.shape
    bpr = base3_bytes_per_row(k)
    t = np.zeros((n, bpr * TRITS_PER_BYTE), dtype=np.int64)
    t[:, :k] = np.where(c < 0, 2, c)
    t = t.reshape(n, bpr, TRITS_PER_BYTE)
    out = np.zeros((n, bpr), dtype=np.int64)
    for d in range(TRITS_PER_BYTE):
        out += t[:, :, d] * 3 ** d
    return out.astype(np.uint8)


def unpack_base3(data, k_eff: int):
    """Inverse of :func:`pack_base3`: (codes (N, K_eff) int8, number of
    invalid bytes).  A byte above 242 has no 5-trit reading; it is counted
    and its 5 codes read as 0."""
    b = np.asarray(data, dtype=np.int64)
    bad = b > 242
    v = np.where(bad, 0, b)
    trits = np.zeros(b.shape + (TRITS_PER_BYTE,), dtype=np.int64)
    for d in range(TRITS_PER_BYTE):
        trits[..., d] = v % 3
        v //= 3
    codes = np.where(trits == 2, -1, trits).reshape(b.shape[0], -1)[:, :k_eff]
    return codes.astype(np.int8), int(bad.sum())


# --------------------------------------------------------------------------
# GPTQ block compensation (Algorithm 1, outer loop with the inverse Hessian)
# --------------------------------------------------------------------------
def gptq_hessian(X, damp_rel: float = 0.01) -> np.ndarray:
    """``H = 2 X^T X + lambda I`` (fp64, K x K) from calibration activations
    ``X`` (tokens x K), the Hessian of Algorithm 1's caption, with the
    dampening ``lambda = damp_rel * mean(diag(2 X^T X))``."""
    X = np.asarray(X, dtype=np.float64)
    h = 2.0 * (X.T @ X)
    lam = damp_rel * float(np.mean(np.diag(h)))
    return h + lam * np.eye(h.shape[0])


def gptq_factor(H) -> np.ndarray:
    """Algorithm 1's first step: ``U = Cholesky(H^-1)^T`` (fp64, upper
    triangular, positive diagonal), so that ``U^T U = H^-1``."""
    P = np.linalg.inv(np.asarray(H, dtype=np.float64))
    P = 0.5 * (P + P.T)
    return np.linalg.cholesky(P).T


# Grid of the fp32 G used by the GPTQ reconstruction (see decode_table32).
GPTQ_G_GRID = 2.0 ** -30


def decode_table32(block: int, n_b: int, signs=None, hadamard: bool = True) -> np.ndarray:
    """``G`` for the GPTQ block reconstruction (n_b x B, fp32): the fp64 table
    rounded to the nearest multiple of 2^-30 (ties to even), then to fp32.

    Entries of G that come out of cancellations (~1e-9) carry fp64 errors
    that are a sizeable part of their fp32 unit in the last place, so two
    correct fp64 evaluations can round them to different fp32 values; the
    absolute grid (far coarser than the fp64 error, finer than fp32's
    resolution at the table's scale) makes the fp32 table a function of the
    real table only, as the zero flush does for A_enc."""
    g = decode_table(block, n_b, signs, hadamard)
    return (np.round(g / GPTQ_G_GRID) * GPTQ_G_GRID).astype(np.float32)


def encode_gptq(W, U, block: int, n_b: int, quantizer: int = TERNARY,
                alpha_mode: int = ALPHA_MAXABS, signs=None, hadamard: bool = True,
                trace: bool = False):
    """Canonical fp32 SDQ encoder with GPTQ block compensation (Algorithm 1).

    ``U``: the upper-triangular factor of ``H^-1`` (``U^T U = H^-1``), used in
    fp32.  Blocks of B columns are taken in order; for block b (columns F,
    later columns R):

    1. codes ``c`` = SDQuant of the current weights of F (canonical upsample
       and eq. (8) scan, as :func:`encode`), with the per-row alpha of the
       ORIGINAL weights (it must be known before the first block's scan);
    2. ``Q = alpha * (c . G)``: the block's reconstruction (Algorithm 1's
       ``SDQuant(W Had, OSR) Had^T``), ``s = sum_j c_j G[j, :]`` summed in
       ascending j from +0, then ``Q = fl(alpha s)``;
    3. ``E = W_F - Q``;
    4. the block's error normalised by the diagonal block of the factor,
       ``E~ = E U_FF^-1`` (forward substitution, ascending column l:
       ``E~_l = t_l / U_ll``, then ``t_k -= E~_l U_lk`` for k > l);
    5. ``W_R -= E~ U_FR`` (per element ``acc = sum_k fl(E~_k U_kj)`` in
       ascending k, then ``W = fl(W - acc)``).

    Step 4 is the reading of Algorithm 1's update ``W_R -= E H^-1_{F,R}``
    (with ``H^-1`` replaced by its Cholesky factor) as the exact block
    update of GPTQ / optimal brain surgeon: for one column it is GPTQ's
    division by the diagonal, and for a block it makes the update equal to
    ``E H_FR H_RR^-1`` (the minimiser of the layer-output error over the
    later columns given the block's error), independent of H's scale.
    Every operation is a rounded fp32 operation in the order stated (numpy
    float32 elementwise ops never fuse a multiply-add).

    Returns ``(codes, alpha)`` as :func:`encode`; with ``trace`` also a list
    of per-block dicts (``E``, ``Et``, ``W_before``, ``W_after`` of the
    later columns, fp32).
    """
    a32 = encode_table(block, n_b, signs, hadamard)
    g32 = decode_table32(block, n_b, signs, hadamard)
    Wc = np.array(W, dtype=np.float32, copy=True)
    U32 = np.asarray(U, dtype=np.float32)
    n, k = Wc.shape
    if k % block or U32.shape != (k, k):
        raise ValueError("W must be N x K with K a multiple of B, U K x K")
    nblk = k // block
    alpha = row_alpha(upsample_canonical(Wc, a32), alpha_mode)
    codes = np.zeros((n, nblk * n_b), dtype=np.int8)
    steps = []
    for b in range(nblk):
        f0, f1 = b * block, (b + 1) * block
        x = upsample_canonical(Wc[:, f0:f1], a32)
        c = sigma_delta_scan(x, alpha, quantizer)[:, 0, :]
        codes[:, b * n_b:(b + 1) * n_b] = c
        cf = c.astype(np.float32)
        s = np.zeros((n, block), dtype=np.float32)
        for j in range(n_b):
            s = s + cf[:, j:j + 1] * g32[j, :]
        q = alpha[:, None] * s
        e = Wc[:, f0:f1] - q
        if f1 == k:
            break
        uff = U32[f0:f1, f0:f1]
        t = e.copy()
        et = np.zeros_like(e)
        for l in range(block):
            et[:, l] = t[:, l] / uff[l, l]
            t[:, l + 1:] = t[:, l + 1:] - et[:, l:l + 1] * uff[l, l + 1:]
        ufr = U32[f0:f1, f1:]
        acc = et[:, 0:1] * ufr[0, :]
        for kk in range(1, block):
            acc = acc + et[:, kk:kk + 1] * ufr[kk, :]
        before = Wc[:, f1:].copy()
        Wc[:, f1:] = Wc[:, f1:] - acc
        assert Wc.dtype == np.float32
        if trace:
            steps.append({"E": e, "Et": et, "W_before": before, "W_after": Wc[:, f1:].copy()})
    return (codes, alpha, steps) if trace else (codes, alpha)
