"""GPU parity: the CUDA path against the oracle on the same seeded inputs.

Codes, alpha and packed layouts must be bit-exact.  Layer outputs must be
within max |y - y_ref| / max |y_ref| <= 1e-2 of the oracle's fp64 forward on
the same codes (the accuracy bar for layer outputs), and every element
within the bound of the path's own arithmetic (tests/errbound.py: T e2m1
terms per 32-code group on the decode path, one bf16 rounding of x_tilde on
the prefill path, fp32 accumulation on both); the element-wise error
max |d| / max(|y_ref|, 1e-3 max |y_ref|) is reported beside it.
"""
from fractions import Fraction

import numpy as np
import pytest

import errbound as EB
import oracle as O
from paper_2510_03275_gb300 import workloads as W

pytestmark = pytest.mark.gpu

TOL = 1e-2


@pytest.fixture(scope="module")
def torch_cuda():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch


def _u32(torch, a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.uint32).view(np.int32)).cuda()


def _np_u32(t):
    return t.cpu().numpy().view(np.uint32)


def _bf16(torch, bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def _desc(sdq, n, k, b, osr, q, had=1, am=0):
    return sdq.LayerDesc(n, k, b, Fraction(osr), q, had, am)


def _encode_compare(sdq, torch, w, block, osr, q, am, had, signs):
    n, k = w.shape
    d = _desc(sdq, n, k, block, osr, q, had, am)
    plan = sdq.Plan(d, signs if had else None)
    codes, alpha = plan.encode(torch.from_numpy(w).cuda())
    torch.cuda.synchronize()
    oc, oa = O.encode(w, block, d.n_b, q, am, signs if had else None, bool(had))
    want = O.pack_plain(oc, q)
    got = _np_u32(codes).reshape(n, -1)
    assert np.array_equal(alpha.cpu().numpy(), oa), "alpha differs"
    mism = np.mean(got != want)
    assert mism == 0.0, f"code word mismatch rate {mism}"
    return plan, codes, alpha, oc, oa


# ---------------------------------------------------------------- encoder
@pytest.mark.parametrize("q", [O.TERNARY, O.BINARY])
@pytest.mark.parametrize("am", [O.ALPHA_MAXABS, O.ALPHA_MEANABS])
@pytest.mark.parametrize("shape", [(17, 20, 4, Fraction(5, 2)), (40, 256, 128, Fraction(3, 2)),
                                   (9, 64, 32, Fraction(3)), (33, 384, 128, Fraction(5, 2))])
@pytest.mark.parametrize("had", [1, 0])
def test_encode_small_bit_exact(sdq, torch_cuda, q, am, shape, had):
    n, k, b, osr = shape
    rng = np.random.default_rng(n * 1000 + k + b)
    w = (rng.standard_normal((n, k)) * 0.02).astype(np.float32)
    signs = np.where(rng.random(b) < 0.5, -1, 1).astype(np.int8)
    _encode_compare(sdq, torch_cuda, w, b, osr, q, am, had, signs)


def test_encode_worked_rows(sdq, torch_cuda, golden):
    """The hand-worked rows, including the OSR 2.5 threshold tie."""
    for key, osr in (("osr2_hadamard4", 2), ("osr25_hadamard4", Fraction(5, 2))):
        g = golden[key]
        w = np.array([g["w"]], dtype=np.float32)
        for q in (O.TERNARY, O.BINARY):
            _, _, _, oc, _ = _encode_compare(sdq, torch_cuda, w, 4, osr, q, 0, 1,
                                             np.array(g["signs"], dtype=np.int8))
            if key == "osr2_hadamard4":
                assert list(oc[0]) == g[("ternary" if q == O.TERNARY else "binary") + "_codes"]
    g = golden["osr1_hadamard_off"]
    w = np.array([g["w"]], dtype=np.float32)
    _, _, _, oc, _ = _encode_compare(sdq, torch_cuda, w, 4, 1, O.TERNARY, 0, 0, None)
    assert list(oc[0]) == g["maxabs"]["ternary_codes"]


@pytest.mark.parametrize("ci", [0, 1])
def test_encode_configs_bit_exact(sdq, torch_cuda, ci):
    """configs 0 and 1 in full: every code and every alpha bit-exact."""
    cfg = W.config(ci)
    for lin in cfg.linears:
        w = W.weights(lin)
        signs = W.hadamard_signs(lin, cfg.block)
        _encode_compare(sdq, torch_cuda, w, cfg.block, lin.osr, cfg.quantizer, 0, 1, signs)


@pytest.mark.parametrize("ci,names", [(2, ("q", "gate", "down")), (3, ("l0.q", "l1.down", "l2.gate", "l3.k")),
                                      (4, ("q", "k", "gate", "down"))])
def test_encode_large_sampled_rows(sdq, torch_cuda, ci, names):
    """Full-size layers encoded on the GPU; the oracle re-encodes a seeded
    sample of rows from the same (device-drawn) weights."""
    from paper_2510_03275_gb300.multiosr import allocate
    torch = torch_cuda
    cfg = W.config(ci, multiosr=allocate)
    for lin in cfg.linears:
        if lin.name not in names:
            continue
        wd = W.weights_device(lin)
        signs = W.hadamard_signs(lin, cfg.block)
        d = _desc(sdq, lin.n_out, lin.k_in, cfg.block, lin.osr, cfg.quantizer)
        plan = sdq.Plan(d, signs)
        codes, alpha = plan.encode(wd)
        rows = np.sort(np.random.default_rng(lin.seed).choice(lin.n_out, 24, replace=False))
        w_rows = wd[torch.as_tensor(rows, device="cuda")].cpu().numpy()
        oc, oa = O.encode(w_rows, cfg.block, d.n_b, cfg.quantizer, 0, signs)
        got = _np_u32(codes).reshape(lin.n_out, -1)[rows]
        assert np.array_equal(alpha.cpu().numpy()[rows], oa)
        assert np.mean(got != O.pack_plain(oc, cfg.quantizer)) == 0.0
        del wd, codes, alpha, plan
        torch.cuda.empty_cache()


# ---------------------------------------------------------------- packing
@pytest.mark.parametrize("q", [O.TERNARY, O.BINARY])
@pytest.mark.parametrize("n,keff", [(16, 128), (33, 300), (17, 50), (5, 1000), (48, 512)])
def test_pack_unpack_bit_exact(sdq, torch_cuda, q, n, keff):
    torch = torch_cuda
    # a descriptor with this K_eff: B = 2 * keff / gcd ... use OSR 1 and B | K
    b = 2
    while keff % (b * 2) == 0 and b < 1024:
        b *= 2
    d = _desc(sdq, n, keff, b, 1, q)
    assert sdq.sdq_k_eff(d) == keff
    plan = sdq.Plan(d)
    codes = W.random_codes(n, keff, q, seed=n + keff)
    plain = O.pack_plain(codes, q).ravel()
    tiled = plan.pack(_u32(torch, plain))
    assert np.array_equal(_np_u32(tiled), O.pack_tiled(codes, q))
    back = plan.alloc_plain()
    bad = torch.zeros(1, dtype=torch.int32, device="cuda")
    sdq.sdq_unpack(plan.handle, tiled, back, bad)
    assert np.array_equal(_np_u32(back), plain)
    assert int(bad.item()) == 0
    if q == O.TERNARY:
        tw = _np_u32(tiled).copy()
        # one invalid field "10" at field 3 of word 0: row 0, k = 3 (never padding)
        tw[0] = (tw[0] & ~np.uint32(0xC0)) | np.uint32(0x80)
        bad.zero_()
        sdq.sdq_unpack(plan.handle, _u32(torch, tw), back, bad)
        torch.cuda.synchronize()
        assert int(bad.item()) == 1


def test_pack_full_size_sampled_tiles(sdq, torch_cuda):
    """llama-70b-layer gate (28672 x 16384 codes): round trip, and a seeded sample of
    (tile, k group) slabs compared with the oracle's tiled layout of the same
    128 rows."""
    torch = torch_cuda
    n, keff = 28672, 16384
    d = _desc(sdq, n, 8192, 128, 2, O.TERNARY)
    plan = sdq.Plan(d)
    g = torch.Generator(device="cuda")
    g.manual_seed(5)
    plain = torch.randint(-2**31, 2**31 - 1, (sdq.sdq_plain_bytes(d) // 4,), generator=g,
                          device="cuda", dtype=torch.int32)
    # ternary words must not contain the invalid pattern 10: map 10 -> 11
    hi = plain & -1431655766                      # 0xAAAAAAAA as int32
    plain = plain | ((hi >> 1) & 0x55555555)
    tiled = plan.pack(plain)
    back = plan.alloc_plain()
    sdq.sdq_unpack(plan.handle, tiled, back)
    assert torch.equal(back, plain)
    pw = plain.cpu().numpy().view(np.uint32).reshape(n, -1)
    nt, ng, wpg = O.tiled_geometry(n, keff, O.TERNARY)
    slabs = _np_u32(tiled).reshape(nt, ng, 128 * wpg)
    rng = np.random.default_rng(1)
    for T in rng.choice(nt, 3, replace=False):
        c = O.unpack_plain(pw[128 * T:128 * T + 128], O.TERNARY, keff)
        for G in rng.choice(ng, 2, replace=False):
            want = O.pack_tiled(c[:, 64 * G:64 * G + 64], O.TERNARY)[:128 * wpg]
            assert np.array_equal(slabs[T, G], want), (T, G)


# ---------------------------------------------------------------- forward
def _setup_layer(sdq, torch, n, k, b, osr, q, seed, codes=None, had=1, rows=None):
    """Plan + packed codes.  With ``rows`` only those rows carry (random)
    codes and every other row is zero, so full-size layers need no
    full-size host arrays."""
    d = _desc(sdq, n, k, b, osr, q, had)
    rng = np.random.default_rng(seed)
    signs = np.where(rng.random(b) < 0.5, -1, 1).astype(np.int8)
    plan = sdq.Plan(d, signs if had else None)
    keff = sdq.sdq_k_eff(d)
    alpha = (rng.random(n) * 0.05 + 0.01).astype(np.float32)
    if rows is None:
        if codes is None:
            codes = W.random_codes(n, keff, q, seed)
        plain_t = _u32(torch, O.pack_plain(codes, q).ravel())
    else:
        codes = W.random_codes(len(rows), keff, q, seed)
        plain_t = torch.zeros(sdq.sdq_plain_bytes(d) // 4, dtype=torch.int32, device="cuda")
        wpr = O.plain_words_per_row(keff, q)
        sub = _u32(torch, O.pack_plain(codes, q))
        plain_t.view(n, wpr)[torch.as_tensor(rows, device="cuda")] = sub
    tiled = plan.pack(plain_t)
    return plan, d, signs if had else None, codes, alpha, tiled


def _x(torch, m, k, seed):
    bits = W.float_to_bf16(np.random.default_rng(seed).standard_normal((m, k)).astype(np.float32))
    return bits, _bf16(torch, bits)


def test_prep_matches_oracle(sdq, torch_cuda):
    torch = torch_cuda
    for (n, k, b, osr, m) in [(16, 512, 128, 2, 1), (16, 768, 128, Fraction(5, 2), 5),
                              (16, 20, 4, Fraction(5, 2), 3), (16, 512, 512, 2, 2)]:
        plan, d, signs, _, _, _ = _setup_layer(sdq, torch, n, k, b, osr, 2, seed=k + m)
        bits, x = _x(torch, m, k, seed=m)
        ws = plan.alloc_workspace(m)
        sdq.sdq_prep_activations(plan.handle, x, m, ws)
        out = torch.empty((m, plan.k_eff), dtype=torch.float32, device="cuda")
        sdq.sdq_read_prep(plan.handle, m, ws, out)
        want = O.prep_activations(W.bf16_to_float(bits), b, d.n_b, signs)
        err = np.abs(out.cpu().numpy() - want).max() / np.abs(want).max()
        assert err < 2e-5, err


def _terms(sdq, d, m):
    import torch
    if m > 64:
        return None   # the prefill path: x_tilde in bf16
    return sdq.sdq_decode_launch_shape(d, m, torch.cuda.get_device_properties(0).multi_processor_count)["T"]


def _check_forward(plan, d, signs, codes, alpha, tiled, sdq, torch, m, seed, rows=None):
    """codes: all rows, or (with ``rows``) just the sampled rows.  Asserts
    every element within its bound; returns max |d| / max |y_ref|."""
    bits, x = _x(torch, m, d.k_in, seed)
    ws = plan.alloc_workspace(m)
    y = plan.forward(tiled, torch.from_numpy(alpha).cuda(), x, ws=ws)
    assert sdq.sdq_workspace_status(plan.handle, m, ws) == 0
    a = alpha if rows is None else alpha[rows]
    xf = W.bf16_to_float(bits)
    yr = O.forward_code_domain(xf, codes, a, d.block, d.n_b, signs)
    yg = y.cpu().numpy()
    if rows is not None:
        yg = yg[:, rows]
    dense = sdq.sdq_forward_route(plan.handle, m) == 3
    EB.check(yg, yr, EB.forward_bound(xf, codes, a, d.block, d.n_b, signs, T=_terms(sdq, d, m), dense=dense),
             f"M={m} n={d.n_out} k={d.k_in} B={d.block} OSR={d.osr}" + (" dense" if dense else ""))
    return np.abs(yg - yr).max() / np.abs(yr).max()


@pytest.mark.parametrize("q", [O.TERNARY, O.BINARY])
@pytest.mark.parametrize("m", [1, 2, 3, 4, 5, 8, 16, 17, 33, 64])
@pytest.mark.parametrize("shape", [(33, 384, 128, Fraction(5, 2)), (256, 512, 512, 2),
                                   (100, 1024, 128, Fraction(3, 2)), (17, 20, 4, Fraction(5, 2)),
                                   (150, 640, 128, 3), (260, 1536, 128, 3)])
def test_forward_decode_small(sdq, torch_cuda, q, m, shape):
    n, k, b, osr = shape
    lay = _setup_layer(sdq, torch_cuda, n, k, b, osr, q, seed=n + k + m)
    err = _check_forward(*lay, sdq, torch_cuda, m, seed=m)
    assert err <= TOL, err


def test_forward_encoded_single_and_opt125m(sdq, torch_cuda):
    """End to end: GPU encode -> pack -> forward vs the oracle's encode and
    fp64 dense forward x . W_hat^T on configs 0 and 1."""
    torch = torch_cuda
    for ci in (0, 1):
        cfg = W.config(ci)
        for lin in cfg.linears[:3]:
            w = W.weights(lin)
            signs = W.hadamard_signs(lin, cfg.block)
            plan, codes, alpha, oc, oa = _encode_compare(sdq, torch, w, cfg.block, lin.osr,
                                                         cfg.quantizer, 0, 1, signs)
            tiled = plan.pack(codes)
            for m in cfg.decode_batches:
                bits = W.activations(lin, m)
                y = plan.forward(tiled, alpha, _bf16(torch, bits)).cpu().numpy()
                w_hat = O.reconstruct(oc, oa, cfg.block, plan.desc.n_b, signs)
                yr = O.forward(W.bf16_to_float(bits), w_hat)
                err = np.abs(y - yr).max() / np.abs(yr).max()
                assert err <= TOL, (ci, lin.name, m, err)


@pytest.mark.parametrize("ci,name", [(2, "q"), (2, "down"), (4, "q"), (4, "k"), (4, "gate"), (4, "down")])
@pytest.mark.parametrize("m", [1, 4, 16, 64])
def test_forward_full_size_sampled(sdq, torch_cuda, ci, name, m):
    """Full-size layers (random seeded codes) in the launch shape the bench
    uses; 48 sampled output rows checked against the oracle."""
    torch = torch_cuda
    cfg = W.config(ci)
    lin = [l for l in cfg.linears if l.name == name][0]
    rows = np.sort(np.random.default_rng(lin.seed + m).choice(lin.n_out, 48, replace=False))
    lay = _setup_layer(sdq, torch, lin.n_out, lin.k_in, cfg.block, lin.osr, cfg.quantizer,
                       seed=lin.seed, rows=rows)
    err = _check_forward(*lay, sdq, torch, m, seed=m + 11, rows=rows)
    assert err <= TOL, err


@pytest.mark.parametrize("name", ["q", "k", "v", "o", "fc1", "fc2"])
@pytest.mark.parametrize("m", [1, 16])
def test_forward_opt125m_all_linears(sdq, torch_cuda, name, m):
    """OPT-125M's six linears (binary codes, OSR 2.5) at M = 1 and 16, every
    output row checked."""
    cfg = W.config(1)
    lin = [l for l in cfg.linears if l.name == name][0]
    lay = _setup_layer(sdq, torch_cuda, lin.n_out, lin.k_in, cfg.block, lin.osr, cfg.quantizer, seed=lin.seed)
    err = _check_forward(*lay, sdq, torch_cuda, m, seed=m + 3)
    assert err <= TOL, err


@pytest.mark.parametrize("name", ["l2.gate", "l3.down", "l0.q"])
def test_forward_llama13b_multiosr_decode(sdq, torch_cuda, name):
    """LLaMA-13B stack under the MultiOSR map, batch-8 decode at full size
    (l2.gate at OSR 3, l3.down at OSR 1.5); 48 sampled rows."""
    from paper_2510_03275_gb300.multiosr import allocate
    torch = torch_cuda
    cfg = W.config(3, multiosr=allocate)
    lin = [l for l in cfg.linears if l.name == name][0]
    if name == "l2.gate":
        assert lin.osr == 3
    if name == "l3.down":
        assert lin.osr == Fraction(3, 2)
    rows = np.sort(np.random.default_rng(lin.seed + 8).choice(lin.n_out, 48, replace=False))
    lay = _setup_layer(sdq, torch, lin.n_out, lin.k_in, cfg.block, lin.osr, cfg.quantizer,
                       seed=lin.seed, rows=rows)
    err = _check_forward(*lay, sdq, torch, 8, seed=19, rows=rows)
    assert err <= TOL, err


def _device_codes(torch, plan, d, q, seed):
    """Random valid plain codes for every row of a full-size layer, drawn on
    the device (torch's seeded generator; ternary fields 00 / 01 / 11 with
    probabilities 1/2, 1/4, 1/4, padding fields zero)."""
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    nw = sdq_plain_words(plan, d)
    w = torch.randint(-2 ** 31, 2 ** 31 - 1, (d.n_out, nw), generator=g, device="cuda", dtype=torch.int64)
    w = w.to(torch.int32)
    if q == O.TERNARY:   # field 10 -> 00: clear the high bit where the low bit is 0
        hi_clear = torch.bitwise_and(torch.bitwise_left_shift(torch.bitwise_not(w), 1), -0x55555556)
        w = torch.bitwise_and(w, torch.bitwise_not(hi_clear))
    keff = plan.k_eff
    per = 32 // q
    full = keff // per
    if full < nw:
        rem = keff - full * per
        if rem:
            w[:, full] = torch.bitwise_and(w[:, full], (1 << (q * rem)) - 1)
            w[:, full + 1:] = 0
        else:
            w[:, full:] = 0
    return w.reshape(-1)


def sdq_plain_words(plan, d):
    return O.plain_words_per_row(plan.k_eff, d.quantizer)


@pytest.mark.parametrize("name,m", [("gate", 1), ("down", 16), ("q", 64)])
def test_forward_full_size_every_row_coded(sdq, torch_cuda, name, m):
    """LLaMA-70B linears with random codes in every row (drawn on the
    device); 64 sampled rows read back, unpacked by the oracle and checked."""
    torch = torch_cuda
    cfg = W.config(4)
    lin = [l for l in cfg.linears if l.name == name][0]
    d = _desc(sdq, lin.n_out, lin.k_in, cfg.block, lin.osr, cfg.quantizer)
    rng = np.random.default_rng(lin.seed)
    signs = np.where(rng.random(cfg.block) < 0.5, -1, 1).astype(np.int8)
    plan = sdq.Plan(d, signs)
    plain = _device_codes(torch, plan, d, cfg.quantizer, seed=lin.seed)
    tiled = plan.pack(plain)
    alpha = (rng.random(lin.n_out) * 0.05 + 0.01).astype(np.float32)
    rows = np.sort(rng.choice(lin.n_out, 64, replace=False))
    wpr = sdq_plain_words(plan, d)
    sub = plain.view(lin.n_out, wpr)[torch.as_tensor(rows, device="cuda")].cpu().numpy().view(np.uint32)
    codes = O.unpack_plain(sub, cfg.quantizer, plan.k_eff)
    err = _check_forward(plan, d, signs, codes, alpha, tiled, sdq, torch, m, seed=m + 23, rows=rows)
    assert err <= TOL, err


def test_workspace_too_small_rejected(sdq, torch_cuda):
    torch = torch_cuda
    plan, d, signs, codes, alpha, tiled = _setup_layer(sdq, torch, 32, 256, 128, 2, 2, seed=3)
    bits, x = _x(torch, 4, 256, 1)
    ws = plan.alloc_workspace(4)
    y = torch.empty((4, 32), device="cuda")
    small = ws[:ws.numel() // 2]
    with pytest.raises(sdq.SdqError) as e:
        sdq.sdq_linear_forward(plan.handle, tiled, torch.from_numpy(alpha).cuda(), x, 4, y, small)
    assert e.value.status == -3


# ---------------------------------------------------------------- prefill
@pytest.mark.parametrize("q", [O.TERNARY, O.BINARY])
@pytest.mark.parametrize("m,shape", [(128, (256, 512, 128, 2)), (200, (300, 384, 128, Fraction(5, 2))),
                                     (65, (17, 20, 4, Fraction(5, 2))), (130, (256, 512, 512, 2)), (130, (150, 640, 128, 3)),
                                     (384, (520, 768, 128, Fraction(3, 2)))])
def test_forward_prefill_small(sdq, torch_cuda, q, m, shape):
    """tcgen05 prefill path (M > 64) against the oracle; x_tilde enters the
    tensor cores as bf16 (one rounding), codes exactly."""
    n, k, b, osr = shape
    lay = _setup_layer(sdq, torch_cuda, n, k, b, osr, q, seed=n + k + m)
    err = _check_forward(*lay, sdq, torch_cuda, m, seed=m)
    assert err <= TOL, err


@pytest.mark.parametrize("q", [O.TERNARY, O.BINARY])
@pytest.mark.parametrize("m,shape", [(768, (300, 512, 128, 2)), (1000, (130, 640, 128, 3)),
                                     (800, (520, 768, 128, Fraction(3, 2)))])
def test_forward_dense_route_small(sdq, torch_cuda, q, m, shape):
    """The dense large-batch route (weights rebuilt in bf16, then one GEMM) on
    ragged rows and batches, OSR 2 / 3 / 1.5, against the oracle within its
    bound."""
    n, k, b, osr = shape
    lay = _setup_layer(sdq, torch_cuda, n, k, b, osr, q, seed=n + k + m)
    assert sdq.sdq_forward_route(lay[0].handle, m) == 3
    err = _check_forward(*lay, sdq, torch_cuda, m, seed=m)
    assert err <= TOL, err


@pytest.mark.parametrize("ci,name,m", [(4, "q", 4096), (4, "gate", 4096), (4, "down", 4096),
                                       (3, "l0.gate", 2048), (3, "l3.down", 2048)])
def test_forward_prefill_full_size_sampled(sdq, torch_cuda, ci, name, m):
    """Full-size prefill in the bench's launch shape; 32 sampled rows."""
    from paper_2510_03275_gb300.multiosr import allocate
    torch = torch_cuda
    cfg = W.config(ci, multiosr=allocate)
    lin = [l for l in cfg.linears if l.name == name][0]
    rows = np.sort(np.random.default_rng(lin.seed + m).choice(lin.n_out, 32, replace=False))
    lay = _setup_layer(sdq, torch, lin.n_out, lin.k_in, cfg.block, lin.osr, cfg.quantizer,
                       seed=lin.seed, rows=rows)
    err = _check_forward(*lay, sdq, torch, m, seed=m + 5, rows=rows)
    assert err <= TOL, err


def test_shared_input_group_constituents(sdq, torch_cuda):
    """One plan over the rows of linears that read one input (q/k/v-shaped:
    256 + 64 + 64 rows of 512 inputs, OSR 2, ternary, q's Hadamard signs):
    every member's codes and alpha equal the oracle's encoding of that member
    alone, bit for bit, and every member's outputs are within their bound at
    M = 1, 8 and 130."""
    torch = torch_cuda
    k = 512
    members = [W.Linear(nm, n, k, Fraction(2), "t5", 0.02, 900 + i)
               for i, (nm, n) in enumerate([("q", 256), ("k", 64), ("v", 64)])]
    ws = [W.weights(l) for l in members]
    signs = W.hadamard_signs(members[0], 128)
    wg = np.concatenate(ws)
    d = _desc(sdq, wg.shape[0], k, 128, 2, O.TERNARY)
    plan = sdq.Plan(d, signs)
    codes, alpha = plan.encode(torch.from_numpy(wg).cuda())
    torch.cuda.synchronize()
    got = _np_u32(codes).reshape(wg.shape[0], -1)
    al = alpha.cpu().numpy()
    r0, per = 0, []
    for l, w in zip(members, ws):
        oc, oa = O.encode(w, 128, d.n_b, O.TERNARY, 0, signs, True)
        assert np.array_equal(al[r0:r0 + l.n_out], oa), l.name
        assert np.array_equal(got[r0:r0 + l.n_out], O.pack_plain(oc, O.TERNARY)), l.name
        per.append(oc)
        r0 += l.n_out
    tiled = plan.pack(codes)
    oc_all = np.concatenate(per)
    for m in (1, 8, 130):
        r0 = 0
        for l in members:
            rows = np.arange(r0, r0 + l.n_out)
            err = _check_forward(plan, d, signs, oc_all[rows], al, tiled, sdq, torch, m, seed=m + 5, rows=rows)
            assert err <= TOL, (l.name, m, err)
            r0 += l.n_out


@pytest.mark.parametrize("group", ["qkv", "gate_up"])
@pytest.mark.parametrize("m", [1, 16])
def test_forward_full_size_shared_input_groups(sdq, torch_cuda, group, m):
    """The LLaMA-70B layer's row-concatenated q/k/v (10240 x 8192) and
    gate/up (57344 x 8192) plans in the bench's launch shape: 16 sampled rows
    of every member checked against the oracle."""
    torch = torch_cuda
    cfg = W.config(4)
    name, members = [g for g in W.shared_input_groups(cfg) if g[0] == group][0]
    n, k = sum(l.n_out for l in members), members[0].k_in
    rng = np.random.default_rng(m + len(members))
    rows, r0 = [], 0
    for l in members:
        rows += list(r0 + rng.choice(l.n_out, 16, replace=False))
        r0 += l.n_out
    rows = np.sort(np.array(rows))
    lay = _setup_layer(sdq, torch, n, k, cfg.block, members[0].osr, cfg.quantizer, seed=members[0].seed, rows=rows)
    err = _check_forward(*lay, sdq, torch, m, seed=m + 31, rows=rows)
    assert err <= TOL, err
