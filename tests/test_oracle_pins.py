"""Pins of the oracle against what the paper and the mathematics fix.

Every test here runs on the CPU.  None of them compares the oracle with
itself: each checks it against a library routine, a closed form, an
algebraic identity of the paper's equations, a hand-worked example
(tests/golden/worked_rows.json) or brute force on tiny inputs.
"""
import math
from fractions import Fraction

import numpy as np
import pytest
import scipy.linalg
import scipy.signal

import oracle as O


# ----------------------------------------------------------------- Hadamard
@pytest.mark.parametrize("n", [1, 2, 4, 8, 16, 32, 64, 128, 256, 512])
def test_sylvester_orthogonality_exact(n):
    """Eq. (13): H H^T = n I, entries +-1 (exact integers)."""
    h = O.sylvester_hadamard(n)
    assert set(np.unique(h)) <= {-1, 1}
    assert np.array_equal(h @ h.T, n * np.eye(n, dtype=np.int64))


@pytest.mark.parametrize("n", [2, 8, 128, 512])
def test_sylvester_matches_library(n):
    """Same matrix as scipy.linalg.hadamard (also Sylvester)."""
    assert np.array_equal(O.sylvester_hadamard(n), scipy.linalg.hadamard(n))


def _fwht(v):
    """Iterative fast Walsh-Hadamard butterflies (independent algorithm)."""
    v = np.array(v, dtype=np.float64)
    h = 1
    while h < v.shape[-1]:
        for i in range(0, v.shape[-1], 2 * h):
            a = v[..., i:i + h].copy()
            b = v[..., i + h:i + 2 * h].copy()
            v[..., i:i + h] = a + b
            v[..., i + h:i + 2 * h] = a - b
        h *= 2
    return v


def test_fwht_equals_dense_product():
    rng = np.random.default_rng(1)
    v = rng.standard_normal((5, 128))
    assert np.allclose(_fwht(v), v @ O.sylvester_hadamard(128), atol=1e-11)


def test_randomised_hadamard_convention_and_orthonormal():
    """Had = diag(d) H / sqrt(B): signs on the input (row) side."""
    had = O.hadamard_matrix(2, signs=[1, -1])
    assert np.allclose(had, np.array([[1, 1], [-1, 1]]) / math.sqrt(2), atol=0)
    rng = np.random.default_rng(2)
    d = np.where(rng.random(128) < 0.5, -1, 1)
    h = O.hadamard_matrix(128, d)
    assert np.abs(h @ h.T - np.eye(128)).max() < 1e-12
    assert np.array_equal(O.hadamard_matrix(8, enabled=False), np.eye(8))


# ----------------------------------------------------------------- Resample
@pytest.mark.parametrize("d", [4, 8, 128, 512])
@pytest.mark.parametrize("osr", [Fraction(3, 2), Fraction(2), Fraction(5, 2), Fraction(3)])
def test_resample_matches_scipy(d, osr):
    """The Resample reading agrees with scipy.signal.resample (up and down)."""
    n_new = int(d * osr)
    rng = np.random.default_rng(d + n_new)
    v = rng.standard_normal((3, d))
    up = O.resample(v, n_new)
    assert np.abs(up - scipy.signal.resample(v, n_new, axis=1)).max() < 1e-12
    u = rng.standard_normal((3, n_new))
    down = O.resample(u, d)
    assert np.abs(down - scipy.signal.resample(u, d, axis=1)).max() < 1e-12


@pytest.mark.parametrize("d,n_new", [(4, 10), (128, 192), (128, 320), (512, 1024), (128, 128)])
def test_resample_down_up_identity(d, n_new):
    rng = np.random.default_rng(7)
    v = rng.standard_normal((4, d))
    assert np.abs(O.resample(O.resample(v, n_new), d) - v).max() < 1e-12


def test_resample_same_length_is_identity():
    v = np.random.default_rng(3).standard_normal((2, 64))
    assert np.abs(O.resample(v, 64) - v).max() < 1e-13


@pytest.mark.parametrize("osr", [2, 3, 4])
def test_resample_integer_osr_interpolates(osr):
    """Band-limited interpolation passes through the original samples."""
    v = np.random.default_rng(osr).standard_normal((3, 32))
    up = O.resample(v, 32 * osr)
    assert np.abs(up[:, ::osr] - v).max() < 1e-12


def test_resample_inband_cosine_closed_form():
    """A cosine below Nyquist maps to the same continuous cosine resampled."""
    d, n_new, f, ph = 16, 40, 3, 0.7
    n = np.arange(d)
    v = np.cos(2 * np.pi * f * n / d + ph)[None]
    m = np.arange(n_new)
    want = np.cos(2 * np.pi * f * m / n_new + ph)
    assert np.abs(O.resample(v, n_new)[0] - want).max() < 1e-12


def test_encode_table_equals_dirichlet_closed_form():
    """A_enc = U Had^T where U[j,k] is the trigonometric-interpolation kernel
    (1/B)[1 + 2 sum_{f=1}^{B/2-1} cos(2 pi f tau) + cos(pi B tau)],
    tau = j/n_b - k/B (the split Nyquist bin), summed directly."""
    B, nb = 8, 20
    d = np.array([1, -1, -1, 1, 1, 1, -1, 1])
    j = np.arange(nb)[:, None]
    k = np.arange(B)[None, :]
    tau = j / nb - k / B
    u = np.ones_like(tau)
    for f in range(1, B // 2):
        u += 2 * np.cos(2 * np.pi * f * tau)
    u += np.cos(np.pi * B * tau)
    u /= B
    had = d[:, None] * scipy.linalg.hadamard(B) / math.sqrt(B)
    want = (u @ had.T).astype(np.float32)
    got = O.encode_table(B, nb, d)
    assert np.abs(got.astype(np.float64) - u @ had.T).max() < 1e-6
    assert np.array_equal(got, want) or np.abs(got - want).max() <= 2 ** -24


def test_encode_table_matches_fft_route():
    """x_up = A_enc w equals Resample(w . Had) computed through the FFT."""
    B, nb = 128, 320
    rng = np.random.default_rng(11)
    d = np.where(rng.random(B) < 0.5, -1, 1)
    w = rng.standard_normal((6, B))
    a = O.encode_table(B, nb, d).astype(np.float64)
    fft_route = O.resample(w @ O.hadamard_matrix(B, d), nb)
    assert np.abs(w @ a.T - fft_route).max() < 1e-5 * np.abs(fft_route).max()


# ------------------------------------------------------------ Sigma-Delta
def test_scan_noise_transfer_identity():
    """Eq. (11): Y = X + (1 - z^-1) E, i.e. y_n - x_n = e_n - e_{n-1} with
    e_n = y_n - i_n and e_0 = 0, sample by sample."""
    rng = np.random.default_rng(5)
    x = rng.uniform(-1, 1, size=(8, 300))
    for qz in (O.TERNARY, O.BINARY):
        _, i, y = O.sigma_delta_scan_f64(x, np.ones((8, 1)), qz)
        e = y - i
        e_prev = np.concatenate([np.zeros((8, 1)), e[:, :-1]], axis=1)
        assert np.abs((y - x) - (e - e_prev)).max() < 1e-12


def test_scan_telescoping():
    """sum_{n<=m} (x_n - y_n) = i_m - y_m."""
    rng = np.random.default_rng(6)
    x = rng.uniform(-0.9, 0.9, size=(4, 200))
    _, i, y = O.sigma_delta_scan_f64(x, np.ones((4, 1)), O.TERNARY)
    assert np.abs(np.cumsum(x - y, axis=1) - (i - y)).max() < 1e-11


@pytest.mark.parametrize("qz,bound", [(O.TERNARY, 0.5), (O.BINARY, 1.0)])
def test_scan_invariant_bounded(qz, bound):
    """With |x| <= alpha the running error |i_n - y_n| stays <= alpha/2
    (ternary) or <= alpha (binary): fp64 reading and canonical fp32."""
    rng = np.random.default_rng(8)
    alpha = 0.37
    x = rng.uniform(-alpha, alpha, size=(16, 1, 512))
    _, i, y = O.sigma_delta_scan_f64(x[:, 0], np.full((16, 1), alpha), qz)
    assert np.abs(i - y).max() <= bound * alpha + 1e-12
    x32 = x.astype(np.float32)
    a32 = np.full(16, alpha, dtype=np.float32)
    codes, st = O.sigma_delta_scan(x32, a32, qz, return_state=True)
    err = st.astype(np.float64) - codes.astype(np.float64) * np.float64(a32[0])
    assert np.abs(err).max() <= bound * alpha * (1 + 1e-5)


def test_scan_constant_input_mean():
    """Constant input c: mean of y over n samples is within alpha/(2n) of c."""
    c, alpha, n = 0.3, 1.0, 400
    _, _, y = O.sigma_delta_scan_f64(np.full((1, n), c), np.ones((1, 1)), O.TERNARY)
    for m in (10, 50, 400):
        assert abs(y[0, :m].mean() - c) <= alpha / (2 * m) + 1e-12


def _frac_scan(x32, alpha32, ternary):
    """Brute force: the scan with exact rationals, rounding every operation
    to fp32 by hand (fp32 add/sub are correctly rounded)."""
    def r32(q):
        return Fraction(float(np.float32(float(q)))) if abs(q) < 2 ** 100 else q
    a = Fraction(float(alpha32))
    i = Fraction(0)
    yp = Fraction(0)
    out = []
    for xv in x32:
        i = r32(i + Fraction(float(xv)))
        i = r32(i - yp)
        if ternary:
            q = 1 if i > a / 2 else (-1 if i < -a / 2 else 0)
        else:
            q = 1 if i >= 0 else -1
        out.append(q)
        yp = q * a
    return out


def test_scan_fp32_matches_rational_brute_force():
    rng = np.random.default_rng(9)
    x = rng.uniform(-1, 1, size=(3, 1, 64)).astype(np.float32)
    a = np.abs(x).reshape(3, -1).max(axis=1).astype(np.float32)
    for qz in (O.TERNARY, O.BINARY):
        codes = O.sigma_delta_scan(x, a, qz)
        for r in range(3):
            assert list(codes[r, 0]) == _frac_scan(x[r, 0], a[r], qz == O.TERNARY)


# ----------------------------------------------------------- worked rows
def test_worked_row_osr1(golden):
    g = golden["osr1_hadamard_off"]
    w = np.array([g["w"]], dtype=np.float32)
    for qz, key in ((O.TERNARY, "ternary"), (O.BINARY, "binary")):
        codes, alpha = O.encode(w, 4, 4, qz, O.ALPHA_MAXABS, hadamard=False)
        assert alpha[0] == g["maxabs"]["alpha"]
        assert list(codes[0]) == g["maxabs"][key + "_codes"]
        x = np.array(g["x_up"], dtype=np.float32).reshape(1, 1, 4)
        c, st = O.sigma_delta_scan(x, alpha, qz, return_state=True)
        assert list((st[0, 0] - c[0, 0] * alpha[0]).astype(float)) == \
            g["maxabs"][key + "_state_i_minus_y"]
    codes, alpha = O.encode(w, 4, 4, O.TERNARY, O.ALPHA_MEANABS, hadamard=False)
    assert alpha[0] == g["meanabs"]["alpha"]
    assert list(codes[0]) == g["meanabs"]["ternary_codes"]
    x = np.array(g["x_up"], dtype=np.float32).reshape(1, 1, 4)
    c, st = O.sigma_delta_scan(x, alpha, O.TERNARY, return_state=True)
    assert list((st[0, 0] - c[0, 0] * alpha[0]).astype(float)) == \
        g["meanabs"]["ternary_state_i_minus_y"]


def test_worked_row_osr2(golden):
    g = golden["osr2_hadamard4"]
    w = np.array([g["w"]], dtype=np.float32)
    x_up = O.upsample_canonical(w, O.encode_table(4, 8, g["signs"]))
    assert np.abs(x_up[0, 0] - np.array(g["x_up"])).max() < 1e-7
    for qz, key in ((O.TERNARY, "ternary"), (O.BINARY, "binary")):
        codes, alpha = O.encode(w, 4, 8, qz, O.ALPHA_MAXABS, g["signs"])
        assert abs(alpha[0] - g["alpha"]) < 1e-7
        assert list(codes[0]) == g[key + "_codes"]
        c64, a64 = O.encode_f64(w, 4, 8, qz, O.ALPHA_MAXABS, g["signs"])
        assert list(c64[0]) == g[key + "_codes"]
        w_hat = O.reconstruct(c64, a64, 4, 8, g["signs"])
        assert np.abs(w_hat[0] - np.array(g["w_hat_" + key])).max() < 1e-12
    # the forward through the code domain returns x . w exactly
    x = np.array([[0.5, -2.0, 3.0, 1.25]])
    y = O.forward_code_domain(x, c64, a64, 4, 8, g["signs"])
    assert abs(y[0, 0] - (-2.0)) < 1e-12


def test_worked_row_osr25_tie(golden):
    """OSR 2.5: canonical x_up equals fp32(0.5 cos(0.4 pi n)) (closed form),
    and the codes equal the rational brute-force fp32 scan on those values."""
    g = golden["osr25_hadamard4"]
    w = np.array([g["w"]], dtype=np.float32)
    a32 = O.encode_table(4, 10, g["signs"])
    x_up = O.upsample_canonical(w, a32)[0, 0]
    closed = np.array([0.5 * math.cos(0.4 * math.pi * n) for n in range(10)], dtype=np.float32)
    assert np.array_equal(x_up, closed)
    for qz in (O.TERNARY, O.BINARY):
        codes, alpha = O.encode(w, 4, 10, qz, O.ALPHA_MAXABS, g["signs"])
        assert alpha[0] == np.float32(g["alpha"])
        assert list(codes[0]) == _frac_scan(closed, alpha[0], qz == O.TERNARY)
    # real arithmetic reaches -theta exactly at n = 2 (0-based):
    i3 = Fraction(1, 2) * 0 + (0.5 * math.cos(0.4 * math.pi) + 0.5 * math.cos(0.8 * math.pi))
    assert abs(float(i3) + 0.25) < 1e-15


# ----------------------------------------------- reconstruction / forward
def _rel_fro(w, w_hat):
    return np.linalg.norm(w - w_hat) / np.linalg.norm(w)


@pytest.mark.parametrize("qz", [O.TERNARY, O.BINARY])
def test_error_decreases_with_osr(qz):
    """Reconstruction error falls strictly as OSR grows (MAXABS alpha)."""
    rng = np.random.default_rng(12)
    B = 128
    d = np.where(rng.random(B) < 0.5, -1, 1)
    w = (rng.standard_normal((48, 512)) * 0.02).astype(np.float32)
    errs = []
    for osr in (Fraction(1), Fraction(3, 2), Fraction(2), Fraction(5, 2), Fraction(3), Fraction(4)):
        nb = int(B * osr)
        codes, alpha = O.encode(w, B, nb, qz, O.ALPHA_MAXABS, d)
        errs.append(_rel_fro(w.astype(np.float64), O.reconstruct(codes, alpha, B, nb, d)))
    assert all(a > b for a, b in zip(errs, errs[1:])), errs
    assert errs[-1] < 0.45


@pytest.mark.parametrize("qz", [O.TERNARY, O.BINARY])
@pytest.mark.parametrize("had", [True, False])
@pytest.mark.parametrize("B,nb", [(128, 320), (16, 24), (64, 64)])
def test_forward_code_domain_identity(qz, had, B, nb):
    """alpha C G x == x W_hat^T (closed-form adjoint identity, fp64), for both
    quantizers, with and without the rotation, at OSR 2.5, 1.5 and 1."""
    rng = np.random.default_rng(13 + B + nb + qz + int(had))
    d = np.where(rng.random(B) < 0.5, -1, 1)
    K = 3 * B
    w = (rng.standard_normal((24, K)) * 0.02).astype(np.float32)
    codes, alpha = O.encode(w, B, nb, qz, O.ALPHA_MAXABS, d, had)
    x = rng.standard_normal((3, K))
    y1 = O.forward(x, O.reconstruct(codes, alpha, B, nb, d, had))
    y2 = O.forward_code_domain(x, codes, alpha, B, nb, d, had)
    assert np.abs(y1 - y2).max() < 1e-10 * np.abs(y1).max()


def test_decimation_adjoint_is_upsample_over_osr_plus_rank1():
    """D^T - U/OSR is the rank-1 Nyquist term (1/n_b) cos(pi B j/n_b)(-1)^k."""
    B, nb = 8, 20
    Dt = O.resample_matrix(nb, B)          # row convention: c . Dt, i.e. D^T
    U = O.resample_matrix(B, nb).T         # column convention: x_up = U v
    j = np.arange(nb)[:, None]
    k = np.arange(B)[None, :]
    want = np.cos(np.pi * B * j / nb) * (-1.0) ** k / nb
    assert np.abs(Dt - U * B / nb - want).max() < 1e-13


@pytest.mark.parametrize("B,osr", [(16, Fraction(5, 2)), (128, 2), (128, Fraction(3, 2)), (64, Fraction(9, 4)),
                                   (256, 2), (2, Fraction(3, 2))])
def test_decimation_adjoint_is_polyphase(B, osr):
    """Band-limited resampling commutes with shifts that land on both grids:
    n_b / B = p / q, a cyclic shift of the n_b codes by p is one of the B
    outputs by q, so row r + p m of D^T is row r rolled by q m: D^T is fixed
    by its first p rows (a polyphase structure)."""
    nb = int(B * osr)
    p, q = osr.numerator, osr.denominator
    rng = np.random.default_rng(B + nb)
    v = rng.standard_normal((3, nb))
    lhs = O.resample(np.roll(v, p, axis=1), B)
    rhs = np.roll(O.resample(v, B), q, axis=1)
    assert np.abs(lhs - rhs).max() < 1e-12 * np.abs(rhs).max()
    Dt = O.resample_matrix(nb, B)
    for j in range(nb):
        r, m = j % p, j // p
        assert np.abs(Dt[j] - np.roll(Dt[r], q * m)).max() < 1e-13


def test_canonical_and_f64_encoders_agree():
    """The fp32 canonical encoder and the fp64 FFT reading pick the same codes
    except where an integrator value lands within rounding of a threshold."""
    rng = np.random.default_rng(14)
    B, nb = 128, 256
    d = np.where(rng.random(B) < 0.5, -1, 1)
    w = (rng.standard_normal((32, 256)) * 0.02).astype(np.float32)
    c32, a32 = O.encode(w, B, nb, O.TERNARY, O.ALPHA_MAXABS, d)
    c64, a64 = O.encode_f64(w, B, nb, O.TERNARY, O.ALPHA_MAXABS, d)
    assert np.abs(a32 - a64).max() <= 1e-6 * a64.max()
    assert np.mean(c32 != c64) < 1e-3


def test_compression_ratio_eq14(golden):
    g = golden["compression_ratio"]
    assert round(O.compression_ratio(1.58, 1.5), 4) == g["osr1.5"]
    assert round(O.compression_ratio(1.58, 2.0), 4) == g["osr2"]


# ---------------------------------------------------------------- packing
def test_pack_plain_literal():
    """Ternary fields 00=0, 01=+1, 11=-1 at bit 2j; binary bit j, 1=+1."""
    c = np.array([[1, -1, 0, 1] + [0] * 12 + [-1]], dtype=np.int8)
    w = O.pack_plain(c, O.TERNARY)
    assert w.shape == (1, 4)
    assert int(w[0, 0]) == 0b01_00_11_01
    assert int(w[0, 1]) == 0b11
    b = np.array([[1, -1, -1, 1, 1] + [-1] * 28 + [1]], dtype=np.int8)
    wb = O.pack_plain(b, O.BINARY)
    assert int(wb[0, 0]) == 0b11001 and int(wb[0, 1]) == 0b10
    rng = np.random.default_rng(15)
    for qz in (O.TERNARY, O.BINARY):
        cc = np.where(rng.random((5, 77)) < 0.5, 1, -1).astype(np.int8)
        if qz == O.TERNARY:
            cc[rng.random((5, 77)) < 0.3] = 0
        assert np.array_equal(O.unpack_plain(O.pack_plain(cc, qz), qz, 77), cc)


def test_pack_tiled_hand_positions():
    """Single codes land where the layout's definition puts them."""
    # ternary, 130 x 200 codes: 2 tiles, K padded to 256 -> 4 groups of 64,
    # 4 words per row per group.  Row 129 = (tile 1, r 1), k 83 = (group 1,
    # word 1, field 3); word = 4 * (128 * (1 * 4 + 1) + 1) + 1 = 2565, and
    # -1 is field value 3 at bit 6.
    c = np.zeros((130, 200), dtype=np.int8)
    c[129, 83] = -1
    w = O.pack_tiled(c, O.TERNARY)
    assert w.size == 2 * 4 * 128 * 4
    nz = np.nonzero(w)[0]
    assert list(nz) == [2565] and int(w[2565]) == 3 << 6
    # binary, 5 x 100 codes: 1 tile, K padded to 128 -> 2 groups, 2 words per
    # row per group.  Row 3, k 70 = (group 1, word 0, bit 6); word =
    # 2 * (128 * 1 + 3) = 262.  +1 sets the bit, -1 leaves it clear.
    cb = -np.ones((5, 100), dtype=np.int8)
    cb[3, 70] = 1
    wb = O.pack_tiled(cb, O.BINARY)
    assert wb.size == 1 * 2 * 128 * 2
    nz = np.nonzero(wb)[0]
    assert list(nz) == [262] and int(wb[262]) == 1 << 6
    rng = np.random.default_rng(16)
    cc = np.where(rng.random((20, 300)) < 0.5, 1, -1).astype(np.int8)
    cc[rng.random((20, 300)) < 0.3] = 0
    assert np.array_equal(O.unpack_tiled(O.pack_tiled(cc, O.TERNARY), O.TERNARY, 20, 300), cc)
    cb = np.where(rng.random((7, 333)) < 0.5, 1, -1).astype(np.int8)
    assert np.array_equal(O.unpack_tiled(O.pack_tiled(cb, O.BINARY), O.BINARY, 7, 333), cb)


@pytest.mark.parametrize("q,n,k", [(O.TERNARY, 200, 300), (O.BINARY, 131, 520)])
def test_tiled_is_a_regrouping_of_plain_chunks(q, n, k):
    """Both layouts keep a row's codes in natural order inside 64-code groups,
    so every (tile, group, row) run of the tiled words equals the plain words
    of that row and group (zero past the last row)."""
    rng = np.random.default_rng(17 + q)
    c = np.where(rng.random((n, k)) < 0.5, 1, -1).astype(np.int8)
    if q == O.TERNARY:
        c[rng.random((n, k)) < 0.4] = 0
    plain = O.pack_plain(c, q)
    tiled = O.pack_tiled(c, q)
    nt, ng, wpr = O.tiled_geometry(n, k, q)
    slabs = tiled.reshape(nt, ng, 128, wpr)
    for T in range(nt):
        for G in range(ng):
            for r in range(128):
                row = 128 * T + r
                want = plain[row, wpr * G: wpr * G + wpr] if row < n and wpr * G < plain.shape[1] \
                    else np.zeros(wpr, np.uint32)
                assert np.array_equal(slabs[T, G, r], want), (T, G, r)
