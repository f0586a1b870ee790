"""Host-side checks of the C ABI: no GPU needed (no kernel is launched)."""
import ctypes
import os
import re
from fractions import Fraction

import numpy as np
import scipy.linalg
import pytest

import oracle as O
from paper_2510_03275_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    with open(os.path.join(ROOT, "include", "sdq.h")) as f:
        txt = f.read()
    return sorted(set(re.findall(r"^\s*(?:[\w\s\*]+?)\b(sdq_\w+)\s*\(", txt, re.M)))


def test_exports_every_declared_symbol(sdq):
    names = _declared()
    assert "sdq_linear_forward" in names and "sdq_encode_rows" in names and len(names) >= 15
    L = sdq.lib()
    for n in names:
        assert hasattr(L, n), n


def test_status_strings(sdq):
    for st in range(0, -8, -1):
        s = sdq.sdq_status_string(st)
        assert s.startswith("SDQ_")
    assert "unknown" in sdq.sdq_status_string(-99)


@pytest.mark.parametrize("n,k,b,osr,q,keff,plain,tiled", [
    (256, 512, 512, Fraction(2), 2, 1024, 256 * 64 * 4, 2 * 16 * 128 * 16),
    (768, 768, 128, Fraction(5, 2), 1, 1920, 768 * 60 * 4, 6 * 30 * 128 * 8),
    (17, 20, 4, Fraction(5, 2), 2, 50, 17 * 4 * 4, 1 * 2 * 128 * 16),
])
def test_geometry(sdq, n, k, b, osr, q, keff, plain, tiled):
    d = sdq.LayerDesc(n, k, b, osr, q)
    assert sdq.sdq_k_eff(d) == keff
    assert sdq.sdq_plain_bytes(d) == plain
    assert sdq.sdq_tiled_bytes(d) == tiled
    assert O.plain_words_per_row(keff, q) * 4 * n == plain
    nt, ng, wpg = O.tiled_geometry(n, keff, q)
    assert nt * ng * 128 * wpg * 4 == tiled


@pytest.mark.parametrize("bad", [
    dict(n_out=0), dict(k_in=100), dict(block=96), dict(block=2048), dict(osr=Fraction(1, 2)),
    dict(osr=Fraction(7, 3)), dict(quantizer=3), dict(hadamard=2), dict(alpha_mode=5),
])
def test_invalid_descriptors(sdq, bad):
    base = dict(n_out=64, k_in=256, block=128, osr=Fraction(2), quantizer=2, hadamard=1, alpha_mode=0)
    base.update(bad)
    d = sdq.LayerDesc(**base)
    with pytest.raises(sdq.SdqError) as e:
        sdq.sdq_build_tables(d)
    assert e.value.status == -1
    h = ctypes.c_void_p()
    assert sdq.lib().sdq_plan_create(ctypes.byref(d.c()), None, ctypes.byref(h)) == -1
    assert sdq.sdq_k_eff(d) == 0 and sdq.sdq_plain_bytes(d) == 0


def test_bad_signs_rejected(sdq):
    d = sdq.LayerDesc(16, 8, 8, Fraction(2))
    with pytest.raises(sdq.SdqError):
        sdq.sdq_build_tables(d, np.array([1, -1, 0, 1, 1, 1, 1, 1]))


def test_null_pointers_rejected(sdq):
    L = sdq.lib()
    assert L.sdq_plan_create(None, None, None) == -1
    assert L.sdq_encode_rows(None, None, None, None, None) == -1
    assert L.sdq_linear_forward(None, None, None, None, 1, None, None, 0, None) == -1
    assert L.sdq_workspace_bytes(None, 1) == 0


def _cfg_tables():
    seen = {}
    for ci in range(5):
        cfg = W.config(ci)
        for lin in cfg.linears:
            s = W.hadamard_signs(lin, cfg.block)
            seen[(cfg.block, lin.osr, s.tobytes())] = (cfg.block, lin.osr, s)
    return list(seen.values())


@pytest.mark.parametrize("block,osr,signs", _cfg_tables()[:6] + [(4, Fraction(5, 2), None),
                                                                  (4, Fraction(2), None),
                                                                  (8, Fraction(9, 4), None)])
@pytest.mark.parametrize("had", [1, 0])
def test_tables_match_oracle(sdq, block, osr, signs, had):
    """The library's fp64-built encode table equals the oracle's bit for bit
    (both are the fp32 rounding of the same real table); G within 1e-6."""
    d = sdq.LayerDesc(16, block, block, osr, 2, had)
    a, g = sdq.sdq_build_tables(d, signs)
    nb = d.n_b
    assert np.array_equal(a, O.encode_table(block, nb, signs, bool(had)))
    assert np.abs(g - O.decode_table(block, nb, signs, bool(had))).max() < 1e-6


def _bf16(h):
    return (np.asarray(h, np.uint32) << 16).view(np.float32).astype(np.float64)


@pytest.mark.parametrize("block,osr", [(16, Fraction(5, 2)), (128, Fraction(2)), (128, Fraction(3, 2)),
                                       (64, Fraction(9, 4)), (256, Fraction(2)), (32, Fraction(1))])
@pytest.mark.parametrize("had", [1, 0])
def test_poly_table_matches_oracle(sdq, block, osr, had):
    """The decode kernel's polyphase table of D^T (host-built): its p phase
    rows, each shifted by q m, give every row of the oracle's D^T to bf16
    hi + lo precision; padding is zero; the trailing floats are d_k / sqrt(B)
    (1 without the rotation)."""
    rng = np.random.default_rng(block + 7 * had)
    signs = np.where(rng.random(block) < 0.5, -1, 1).astype(np.int8)
    d = sdq.LayerDesc(16, block, block, osr, 2, had)
    t, p, q = sdq.sdq_build_poly_table(d, signs)
    assert Fraction(p, q) == Fraction(osr)
    st = 2 * block + 8
    assert t.size == 2 * p * st + block
    ent = t[:2 * p * st].reshape(p, st, 2)
    assert not ent[:, 2 * block:, :].any()
    hi, lo = ent[:, :2 * block, 0], ent[:, :2 * block, 1]
    first = _bf16(hi & 0xFFFF) + _bf16(lo & 0xFFFF)     # tap d mod B
    second = _bf16(hi >> 16) + _bf16(lo >> 16)          # tap d + 1 mod B
    Dt = O.resample_matrix(d.n_b, block)                 # D^T, n_b x B
    tol = 2.0 ** -15 * np.abs(Dt).max()
    idx = np.arange(2 * block)
    for r in range(p):
        assert np.abs(first[r] - Dt[r, idx % block]).max() <= tol
        assert np.abs(second[r] - Dt[r, (idx + 1) % block]).max() <= tol
    for j in range(d.n_b):   # every row from its phase: D^T[r + p m][i] = row r at (i - q m) mod B
        r, m = j % p, j // p
        start = (-q * m) % block
        assert np.abs(first[r, start:start + block] - Dt[j, :]).max() <= tol
    scale = t[2 * p * st:].view(np.float32).astype(np.float64)
    want = signs / np.sqrt(block) if had else np.ones(block)
    assert np.abs(scale - want).max() <= 1e-7


@pytest.mark.parametrize("block,osr", [(512, Fraction(2)), (128, Fraction(17, 16)), (8, Fraction(2))])
def test_poly_table_unsupported(sdq, block, osr):
    """No table where the decode kernel streams G instead: B above 256, 17
    phases (more than 16 KB of entries), B not a multiple of 16."""
    d = sdq.LayerDesc(16, block, block, osr, 2, 1)
    with pytest.raises(sdq.SdqError) as e:
        sdq.sdq_build_poly_table(d)
    assert e.value.status == -2   # SDQ_ERR_UNSUPPORTED


def _launch_shapes():
    seen = {}
    for ci in range(5):
        cfg = W.config(ci)
        for lin in cfg.linears:
            seen[(lin.n_out, lin.k_in, cfg.block, Fraction(lin.osr), cfg.quantizer)] = None
    seen[(77, 640, 64, Fraction(9, 4), 2)] = None
    seen[(129, 272, 16, Fraction(5, 2), 1)] = None
    seen[(5, 4096, 1024, Fraction(4), 2)] = None
    return list(seen)


@pytest.mark.parametrize("sms", [152, 148, 132, 20])
def test_decode_launch_shapes_fit(sdq, sms):
    """Every decode launch shape the plan would choose keeps the kernel's
    invariants: at most one CTA per SM, k chunks covering K with none empty,
    a ring of 4..24 stages in multiples of 4, TMEM columns within 512, the
    B operand and ring within the shared-memory limit, stage copies within
    the mbarrier transaction count, and a streamed B operand only past the
    one-kernel route (M > 4)."""
    for n, k, b, osr, qz in _launch_shapes():
        d = sdq.LayerDesc(n, k, b, osr, qz, 1, 0)
        kb = -(-sdq.sdq_k_eff(d) // 128)
        blk = 128 * 128 * qz // 8
        for m in range(1, 65):
            s = sdq.sdq_decode_launch_shape(d, m, sms)
            assert s["T"] == (4 if m <= 8 else 2) and s["NP"] == -(-(m * s["T"]) // 16) * 16
            assert 1 <= s["S"] and 1 <= s["P"] and s["S"] * s["P"] <= sms
            assert (s["S"] - 1) * s["CB"] < kb <= s["S"] * s["CB"]
            assert 4 <= s["ring"] <= 24 and s["ring"] % 4 == 0
            assert 2 * 2 * 32 * s["sb"] + 2 * s["nbuf"] * s["NP"] <= 512
            assert s["streamed"] in (0, 1) and (m > 4 or not s["streamed"])
            assert s["slot_bytes"] == s["sb"] * (blk + (s["NP"] * 128 if s["streamed"] else 0))
            assert s["b_bytes"] == (0 if s["streamed"] else s["CB"] * s["NP"] * 128)
            assert 1024 + s["b_bytes"] + s["ring"] * s["slot_bytes"] <= s["smem"] <= s["smem_limit"]
            assert s["slot_bytes"] < (1 << 20)
            assert max(-(-s["CB"] // s["sb"]), min(2, s["CB"])) <= 128   # stages per row tile


@pytest.mark.parametrize("block,osr", [(128, Fraction(2)), (16, Fraction(5, 2)), (64, Fraction(9, 4))])
@pytest.mark.parametrize("had", [1, 0])
def test_poly_table_gives_x_tilde(sdq, block, osr, had):
    """The decode kernel's order of work, in numpy, with the library's own
    table: scale x by the table's d_k / sqrt(B), a Walsh-Hadamard transform
    (Sylvester order), then D^T from the phase rows and shifts, equals the
    oracle's x_tilde = G x_b (to the bf16 hi + lo precision of the table)."""
    rng = np.random.default_rng(block + had)
    signs = np.where(rng.random(block) < 0.5, -1, 1).astype(np.int8)
    d = sdq.LayerDesc(16, 2 * block, block, osr, 2, had)
    t, p, q = sdq.sdq_build_poly_table(d, signs)
    st, nb = 2 * block + 8, d.n_b
    ent = t[:2 * p * st].reshape(p, st, 2)
    taps = _bf16(ent[:, :block, 0] & 0xFFFF) + _bf16(ent[:, :block, 1] & 0xFFFF)   # D^T[r][0..B)
    scale = t[2 * p * st:].view(np.float32).astype(np.float64)
    x = rng.standard_normal((2, 2 * block)).astype(np.float32).astype(np.float64)
    want = O.prep_activations(x, block, nb, signs, bool(had))
    H = scipy.linalg.hadamard(block).astype(np.float64)
    got = np.zeros_like(want)
    for m in range(2):
        for b in range(2):
            u = x[m, b * block:(b + 1) * block] * scale
            if had:
                u = H @ u
            for j in range(nb):
                r, mm = j % p, j // p
                row = np.roll(taps[r], q * mm)          # D^T[j][i] = D^T[r][(i - q m) mod B]
                got[m, b * nb + j] = row @ u
    assert np.abs(got - want).max() <= 2.0 ** -14 * np.abs(want).max()
