"""Host-side checks of the C ABI: no GPU needed (no kernel is launched)."""
import ctypes
import os
import re
from fractions import Fraction

import numpy as np
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
    # the fp32 G of the GPTQ block reconstruction: the same rounding of the same real table
    assert np.array_equal(sdq.sdq_build_gptq_table(d, signs), O.decode_table32(block, nb, signs, bool(had)))


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
    invariants: at most one CTA per SM (or one per k chunk, where a chunk's
    B operand would not fit otherwise), k chunks covering K with none empty,
    a ring of 4..32 stages in multiples of 4 (one expander set per ring
    slot), 1, 2 or 4 MMA pipelines, TMEM columns within 512 (4 or 8 slots of
    16 sb code columns and their B-scale columns: sb 4-aligned sets, with
    4-column sets rounded up to one 4, 8 or 16-column store, 4 A-scale
    columns, npipe x nbuf accumulators), the B
    image (8 or NP rows per block pair) or the streamed stage slots, its
    scale words and the ring within the shared-memory limit, and
    the e2m1 term count of the batch size."""
    for n, k, b, osr, qz in _launch_shapes():
        d = sdq.LayerDesc(n, k, b, osr, qz, 1, 0)
        kb = -(-sdq.sdq_k_eff(d) // 128)
        blk = 128 * 128 * qz // 8
        for m in range(1, 65):
            s = sdq.sdq_decode_launch_shape(d, m, sms)
            t = 6 if m <= 4 else (4 if m <= 16 else 3)
            assert s["T"] == t and s["NP"] == -(-(m * t) // 16) * 16
            assert 1 <= s["S"] and 1 <= s["P"] and (s["S"] * s["P"] <= sms or s["P"] == 1)
            assert (s["S"] - 1) * s["CB"] < kb <= s["S"] * s["CB"]
            assert 4 <= s["ring"] <= 32 and s["ring"] % 4 == 0
            assert s["npipe"] in (1, 2, 4) and s["nbuf"] in (1, 2) and s["ns"] in (4, 8)
            assert s["ss"] == 4 * (-(-(-(-s["NP"] // 32)) // 4))
            assert 1 <= s["sb"] <= 4
            sss = ({1: 4, 2: 8}.get(s["sb"], 16) if s["ss"] == 4 else s["sb"] * s["ss"])
            assert s["ns"] * (16 * s["sb"] + sss) + 4 + s["npipe"] * s["nbuf"] * s["NP"] <= 512
            n_b = sdq.sdq_k_eff(d) // (k // b)
            if s["bstream"]:
                # B rows and scale words stream with each stage: whole block
                # pairs (even sb, chunks starting on a pair), only where the
                # prepare kernel writes the image, slots 1 KB-aligned
                assert n_b % 64 == 0 and m * t > 8 and s["sb"] % 2 == 0
                assert s["S"] == 1 or s["CB"] % 2 == 0
                bslot = s["sb"] // 2 * s["NP"] * 128 + s["sb"] * s["NP"] * 4
                assert s["slot_bytes"] == -(-(s["sb"] * blk + bslot) // 1024) * 1024
                assert s["b_bytes"] == 0
                assert 1024 + s["ring"] * s["slot_bytes"] <= s["smem"] <= s["smem_limit"]
                npr = -(-s["CB"] // 2)
                assert max(-(-2 * npr // s["sb"]), min(2, npr)) <= 128   # stages per row tile
            else:
                assert s["slot_bytes"] == s["sb"] * blk
                # the image's rows per block pair: the first 8-row group alone
                # when the batch's term rows fit in it and the prepare kernel
                # writes the image (n_b a multiple of 64)
                brow = 8 if (n_b % 64 == 0 and m * t <= 8) else s["NP"]
                assert s["b_bytes"] == (s["CB"] // 2 + 1) * brow * 128
                sfb = -(-(s["CB"] * s["NP"] * 4) // 16) * 16   # the chunk's B scale words
                assert 1024 + s["b_bytes"] + sfb + s["ring"] * s["slot_bytes"] <= s["smem"] <= s["smem_limit"]
                assert max(-(-s["CB"] // s["sb"]), min(2, s["CB"])) <= 128   # stages per row tile


@pytest.mark.parametrize("n,k,osr,q", [(16, 128, Fraction(2), 2), (7, 640, Fraction(17, 16), 2),
                                       (16, 128, Fraction(2), 1)])
def test_base3_bytes_geometry(sdq, n, k, osr, q):
    d = sdq.LayerDesc(n, k, 128, osr, q)
    if q == 1:
        assert sdq.sdq_base3_bytes(d) == 0
    else:
        assert sdq.sdq_base3_bytes(d) == n * O.base3_bytes_per_row(sdq.sdq_k_eff(d))


def test_header_compiles_as_c99(tmp_path):
    """include/sdq.h is a plain C header: no C++ or torch types at the boundary."""
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("gcc not found")
    src = tmp_path / "use.c"
    src.write_text('#include "sdq.h"\nint main(void) { sdq_plan p = 0; (void)p; return 0; }\n')
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    r = subprocess.run([gcc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", "-I", inc, "-c", str(src),
                        "-o", str(tmp_path / "use.o")], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
