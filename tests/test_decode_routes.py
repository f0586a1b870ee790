"""GPU: the two decode routes against the oracle and each other.

sdq_linear_forward runs the prepare kernel (x_tilde, the B operand image and,
with split-K, y cleared) and the contraction, whose split-K partials go into
y by float atomics; sdq_prep_activations + sdq_contract leave y to the
deterministic ticket route (the last CTA of a row tile sums its partials in
k-chunk order).  Both are checked element by element against the oracle
with the bound of the decode arithmetic (tests/errbound.py), on the B operand
image route (n_b a multiple of 64) and the in-kernel term writer (other n_b),
and for their use of the workspace: nothing in it needs to start at zero, and
one workspace may serve several layers in turn.
"""
from fractions import Fraction

import numpy as np
import pytest

import errbound as EB
import oracle as O
from paper_2510_03275_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch_cuda():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch


def _layer(sdq, torch, n, k, b, osr, q, seed, hadamard=1):
    d = sdq.LayerDesc(n, k, b, Fraction(osr), q, hadamard, 0)
    rng = np.random.default_rng(seed)
    signs = np.where(rng.random(b) < 0.5, -1, 1).astype(np.int8)
    plan = sdq.Plan(d, signs if hadamard else None)
    keff = sdq.sdq_k_eff(d)
    codes = W.random_codes(n, keff, q, seed)
    plain = torch.from_numpy(O.pack_plain(codes, q).ravel().view(np.int32)).cuda()
    tiled = plan.pack(plain)
    alpha = (rng.random(n) * 0.05 + 0.01).astype(np.float32)
    return plan, d, signs if hadamard else None, codes, alpha, tiled


def _x(torch, m, k, seed):
    bits = W.float_to_bf16(np.random.default_rng(seed).standard_normal((m, k)).astype(np.float32))
    x = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).cuda()
    return bits, x


def _terms(sdq, d, m):
    import torch
    return sdq.sdq_decode_launch_shape(d, m, torch.cuda.get_device_properties(0).multi_processor_count)["T"]


# Ragged N, K_eff not a multiple of 128 (padding inside the last chunk), OSR
# 2.5 / 1.5 / 3 (128-code blocks straddle input blocks), n_b = 256, 1024, 384
# (the B operand image) and 40, 144, 136, 96 (the in-kernel term writer).
SHAPES = [(33, 384, 128, Fraction(5, 2)), (100, 1024, 128, Fraction(3, 2)),
          (300, 2048, 128, 2), (129, 272, 16, Fraction(5, 2)), (64, 1024, 512, 2),
          (77, 640, 64, Fraction(9, 4)), (70, 512, 128, Fraction(17, 16)), (150, 640, 128, 3),
          (90, 512, 32, 3)]


@pytest.mark.parametrize("q", [O.TERNARY, O.BINARY])
@pytest.mark.parametrize("m", [1, 3, 4, 8, 16, 40, 64])
@pytest.mark.parametrize("shape", SHAPES)
def test_routes_match_oracle_and_each_other(sdq, torch_cuda, q, m, shape):
    torch = torch_cuda
    n, k, b, osr = shape
    plan, d, signs, codes, alpha, tiled = _layer(sdq, torch, n, k, b, osr, q, seed=n + k + 7 * m)
    bits, x = _x(torch, m, k, seed=3 * m + 1)
    al = torch.from_numpy(alpha).cuda()
    assert sdq.sdq_forward_kernels(plan.handle, m, x) == 2
    ws = plan.alloc_workspace(m)
    ws.fill_(0xFF)
    y1 = plan.forward(tiled, al, x, ws=ws)
    assert sdq.sdq_workspace_status(plan.handle, m, ws) == 0
    y2 = torch.full_like(y1, float("nan"))
    sdq.sdq_prep_activations(plan.handle, x, m, ws)
    sdq.sdq_contract(plan.handle, tiled, al, m, y2, ws)
    assert sdq.sdq_workspace_status(plan.handle, m, ws) == 0
    xf = W.bf16_to_float(bits)
    yr = O.forward_code_domain(xf, codes, alpha, b, d.n_b, signs)
    bound = EB.forward_bound(xf, codes, alpha, b, d.n_b, signs, T=_terms(sdq, d, m))
    EB.check(y1.cpu().numpy(), yr, bound, "sdq_linear_forward")
    EB.check(y2.cpu().numpy(), yr, bound, "sdq_contract")
    # the two routes differ only in the order of the split-K sums
    assert np.abs(y1.cpu().numpy() - y2.cpu().numpy()).max() <= 1e-5 * np.abs(yr).max()


@pytest.mark.parametrize("m", [1, 3, 16])
@pytest.mark.parametrize("shape", [(300, 2048, 128, 2), (129, 272, 16, Fraction(5, 2)),
                                   (70, 512, 128, Fraction(17, 16))])
def test_forward_without_hadamard(sdq, torch_cuda, m, shape):
    """Layers encoded without the Hadamard rotation (G = D^T) match the
    oracle on both routes."""
    torch = torch_cuda
    n, k, b, osr = shape
    plan, d, signs, codes, alpha, tiled = _layer(sdq, torch, n, k, b, osr, O.TERNARY, seed=n + m, hadamard=0)
    bits, x = _x(torch, m, k, seed=5 * m + 2)
    y = plan.forward(tiled, torch.from_numpy(alpha).cuda(), x).cpu().numpy()
    xf = W.bf16_to_float(bits)
    yr = O.forward_code_domain(xf, codes, alpha, b, d.n_b, None, hadamard=False)
    EB.check(y, yr, EB.forward_bound(xf, codes, alpha, b, d.n_b, None, T=_terms(sdq, d, m), hadamard=False))


@pytest.mark.parametrize("m", [1, 4])
def test_contract_ignores_workspace_contents(sdq, torch_cuda, m):
    """Split-K tickets and the call record carry the call's tag: random,
    all-ones and stale workspace contents give the same result, bit for bit
    on the deterministic route; the atomic route stays within the bound."""
    torch = torch_cuda
    plan, d, signs, codes, alpha, tiled = _layer(sdq, torch, 1000, 4096, 128, 2, O.TERNARY, seed=5)
    bits, x = _x(torch, m, 4096, seed=9)
    al = torch.from_numpy(alpha).cuda()
    ws = plan.alloc_workspace(m)
    g = torch.Generator(device="cuda")
    g.manual_seed(1)
    xf = W.bf16_to_float(bits)
    yr = O.forward_code_domain(xf, codes, alpha, 128, d.n_b, signs)
    bound = EB.forward_bound(xf, codes, alpha, 128, d.n_b, signs, T=_terms(sdq, d, m))
    outs = []
    for fill in ("random", "ones", "stale", "stale"):
        if fill == "random":
            ws.copy_(torch.randint(0, 256, ws.shape, generator=g, device="cuda", dtype=torch.int32).to(torch.uint8))
        elif fill == "ones":
            ws.fill_(0xFF)
        y = torch.empty((m, 1000), dtype=torch.float32, device="cuda")
        sdq.sdq_prep_activations(plan.handle, x, m, ws)
        sdq.sdq_contract(plan.handle, tiled, al, m, y, ws)
        assert sdq.sdq_workspace_status(plan.handle, m, ws) == 0
        outs.append(y.cpu().numpy())
        y1 = plan.forward(tiled, al, x, ws=ws).cpu().numpy()
        assert sdq.sdq_workspace_status(plan.handle, m, ws) == 0
        EB.check(y1, yr, bound, f"linear_forward after {fill}")
    EB.check(outs[0], yr, bound, "contract")
    for o in outs[1:]:
        assert np.array_equal(o, outs[0])


def test_one_workspace_serves_several_layers(sdq, torch_cuda):
    """Layers with different row-tile counts and split-K grids take turns on
    one workspace (sized for the largest), both routes mixed."""
    torch = torch_cuda
    layers = [_layer(sdq, torch, n, k, 128, 2, O.TERNARY, seed=n) for n, k in
              [(1024, 8192), (4096, 1024), (640, 2048)]]
    ms = [1, 4, 2]
    size = max(sdq.sdq_workspace_bytes(lay[0].handle, m) for lay in layers for m in ms + [8])
    ws = torch.empty(size, dtype=torch.uint8, device="cuda")
    ws.fill_(0x5A)
    for rnd in range(2):
        for i, (plan, d, signs, codes, alpha, tiled) in enumerate(layers):
            m = ms[(i + rnd) % 3] if rnd == 0 else 8
            bits, x = _x(torch, m, d.k_in, seed=17 * i + m)
            al = torch.from_numpy(alpha).cuda()
            if (i + rnd) % 2:
                y = plan.forward(tiled, al, x, ws=ws)
            else:
                y = torch.empty((m, d.n_out), dtype=torch.float32, device="cuda")
                sdq.sdq_prep_activations(plan.handle, x, m, ws)
                sdq.sdq_contract(plan.handle, tiled, al, m, y, ws)
            assert sdq.sdq_workspace_status(plan.handle, m, ws) == 0
            xf = W.bf16_to_float(bits)
            yr = O.forward_code_domain(xf, codes, alpha, 128, d.n_b, signs)
            EB.check(y.cpu().numpy(), yr, EB.forward_bound(xf, codes, alpha, 128, d.n_b, signs,
                                                           T=_terms(sdq, d, m)), f"{rnd} {i} {m}")


@pytest.mark.parametrize("name", ["q", "k", "gate", "down"])
def test_llama70b_decode_kernels(sdq, torch_cuda, name):
    """Every decode call is two kernels: the prepare kernel and the
    contraction."""
    torch = torch_cuda
    cfg = W.config(4)
    lin = [l for l in cfg.linears if l.name == name][0]
    d = sdq.LayerDesc(lin.n_out, lin.k_in, cfg.block, Fraction(lin.osr), cfg.quantizer, 1, 0)
    plan = sdq.Plan(d)
    x = torch.zeros((16, lin.k_in), dtype=torch.bfloat16, device="cuda")
    for m in (1, 8, 16):
        assert sdq.sdq_forward_kernels(plan.handle, m, x) == 2


@pytest.mark.parametrize("m", [1, 4, 16, 64])
@pytest.mark.parametrize("shape", [(300, 2048, 128, 2), (129, 272, 16, Fraction(5, 2)), (1000, 4096, 128, 2)])
def test_contract_add_accumulates(sdq, torch_cuda, m, shape):
    """sdq_contract_add adds the layer's output into y (a residual stream):
    y0 + W_hat x within the bound, twice in a row gives y0 + 2 W_hat x, and
    batches above the decode range are refused."""
    torch = torch_cuda
    n, k, b, osr = shape
    plan, d, signs, codes, alpha, tiled = _layer(sdq, torch, n, k, b, osr, O.TERNARY, seed=n + 3 * m)
    bits, x = _x(torch, m, k, seed=7 * m + 3)
    al = torch.from_numpy(alpha).cuda()
    ws = plan.alloc_workspace(m)
    sdq.sdq_prep_activations(plan.handle, x, m, ws)
    y0 = np.random.default_rng(m + n).standard_normal((m, n)).astype(np.float32)
    y = torch.from_numpy(y0).cuda()
    sdq.sdq_contract_add(plan.handle, tiled, al, m, y, ws)
    assert sdq.sdq_workspace_status(plan.handle, m, ws) == 0
    xf = W.bf16_to_float(bits)
    yr = O.forward_code_domain(xf, codes, alpha, b, d.n_b, signs)
    bound = EB.forward_bound(xf, codes, alpha, b, d.n_b, signs, T=_terms(sdq, d, m))
    # the float adds into y0 round at |y0| (ulp 2^-23 of its magnitude)
    slack = 2.0 ** -22 * (np.abs(y0) + np.abs(yr))
    assert np.all(np.abs(y.cpu().numpy() - y0 - yr) <= bound + slack)
    sdq.sdq_contract_add(plan.handle, tiled, al, m, y, ws)
    assert np.all(np.abs(y.cpu().numpy() - y0 - 2 * yr) <= 2 * bound + 2 * slack)


def test_contract_add_refuses_prefill_batches(sdq, torch_cuda):
    torch = torch_cuda
    plan, d, signs, codes, alpha, tiled = _layer(sdq, torch, 256, 512, 128, 2, O.TERNARY, seed=1)
    m = 128
    ws = plan.alloc_workspace(m)
    y = torch.zeros((m, 256), dtype=torch.float32, device="cuda")
    with pytest.raises(sdq.SdqError) as e:
        sdq.sdq_contract_add(plan.handle, tiled, torch.from_numpy(alpha).cuda(), m, y, ws)
    assert e.value.status == -2   # SDQ_ERR_UNSUPPORTED
