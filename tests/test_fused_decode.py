"""GPU: the single-kernel decode forward (the decode kernel building its own
fp8 B operand from x) against the oracle and against the two-kernel path
(sdq_prep_activations + sdq_contract) on the same inputs, and its use of the
workspace: nothing in it needs to start at zero, and one workspace may serve
several layers in turn.
"""
from fractions import Fraction

import numpy as np
import pytest

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
    plan = sdq.Plan(d, signs)
    keff = sdq.sdq_k_eff(d)
    codes = W.random_codes(n, keff, q, seed)
    plain = torch.from_numpy(O.pack_plain(codes, q).ravel().view(np.int32)).cuda()
    tiled = plan.pack(plain)
    alpha = (rng.random(n) * 0.05 + 0.01).astype(np.float32)
    return plan, d, signs, codes, alpha, tiled


def _x(torch, m, k, seed):
    bits = W.float_to_bf16(np.random.default_rng(seed).standard_normal((m, k)).astype(np.float32))
    x = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).cuda()
    return bits, x


def _rel(a, b):
    return float(np.abs(a - b).max() / np.abs(b).max())


# Shapes the fused path takes: ragged N, K_eff not a multiple of 128 (padding
# inside the last chunk), OSR 2.5 / 1.5 (128-code blocks straddle input
# blocks), B = 16, 64 and 256 (the polyphase build with 1, 2 and 8 inputs per
# lane), and OSR 17/16, whose 17 phases make the polyphase table too large:
# the dense-G build.
FUSED_SHAPES = [(33, 384, 128, Fraction(5, 2)), (100, 1024, 128, Fraction(3, 2)),
                (300, 2048, 128, 2), (129, 272, 16, Fraction(5, 2)), (64, 1024, 256, 2),
                (77, 640, 64, Fraction(9, 4)), (70, 512, 128, Fraction(17, 16))]


@pytest.mark.parametrize("q", [O.TERNARY, O.BINARY])
@pytest.mark.parametrize("m", [1, 2, 3, 4])
@pytest.mark.parametrize("shape", FUSED_SHAPES)
def test_fused_forward_matches_oracle_and_two_kernel_path(sdq, torch_cuda, q, m, shape):
    torch = torch_cuda
    n, k, b, osr = shape
    plan, d, signs, codes, alpha, tiled = _layer(sdq, torch, n, k, b, osr, q, seed=n + k + 7 * m)
    bits, x = _x(torch, m, k, seed=3 * m + 1)
    al = torch.from_numpy(alpha).cuda()
    fused = sdq.sdq_forward_kernels(plan.handle, m, x) == 1
    if m == 1:
        assert fused, "one-kernel forward expected at M = 1 on this shape"
    ws = plan.alloc_workspace(m)
    ws.fill_(0xFF)                      # the fused call must not need (or write) x_tilde
    y1 = plan.forward(tiled, al, x, ws=ws)
    assert sdq.sdq_workspace_status(plan.handle, m, ws) == 0
    xt = torch.empty((m, plan.k_eff), dtype=torch.float32, device="cuda")
    sdq.sdq_read_prep(plan.handle, m, ws, xt)
    assert torch.isnan(xt).all().item() == fused, "x_tilde written iff the two-kernel path ran"
    y2 = torch.empty_like(y1)
    sdq.sdq_prep_activations(plan.handle, x, m, ws)
    sdq.sdq_contract(plan.handle, tiled, al, m, y2, ws)
    assert sdq.sdq_workspace_status(plan.handle, m, ws) == 0
    yr = O.forward_code_domain(W.bf16_to_float(bits), codes, alpha, b, d.n_b, signs)
    e1, e2 = _rel(y1.cpu().numpy(), yr), _rel(y2.cpu().numpy(), yr)
    assert e1 <= 1e-3 and e2 <= 1e-3, (e1, e2)
    assert _rel(y1.cpu().numpy(), y2.cpu().numpy()) <= 1e-3


@pytest.mark.parametrize("m", [1, 3])
@pytest.mark.parametrize("shape", [(300, 2048, 128, 2), (129, 272, 16, Fraction(5, 2)),
                                   (70, 512, 128, Fraction(17, 16))])
def test_fused_forward_without_hadamard(sdq, torch_cuda, m, shape):
    """Layers encoded without the Hadamard rotation (G = D^T): the one-kernel
    build skips the Walsh-Hadamard transform and matches the oracle."""
    torch = torch_cuda
    n, k, b, osr = shape
    plan, d, signs, codes, alpha, tiled = _layer(sdq, torch, n, k, b, osr, O.TERNARY, seed=n + m, hadamard=0)
    bits, x = _x(torch, m, k, seed=5 * m + 2)
    assert sdq.sdq_forward_kernels(plan.handle, m, x) == 1
    y = plan.forward(tiled, torch.from_numpy(alpha).cuda(), x).cpu().numpy()
    yr = O.forward_code_domain(W.bf16_to_float(bits), codes, alpha, b, d.n_b, signs, hadamard=False)
    assert _rel(y, yr) <= 1e-3


def test_fused_forward_ignores_workspace_contents(sdq, torch_cuda):
    """Split-K tickets and the call record carry the call number: random,
    all-ones and stale workspace contents give the same result."""
    torch = torch_cuda
    plan, d, signs, codes, alpha, tiled = _layer(sdq, torch, 1000, 4096, 128, 2, O.TERNARY, seed=5)
    bits, x = _x(torch, 1, 4096, seed=9)
    assert sdq.sdq_forward_kernels(plan.handle, 1, x) == 1
    al = torch.from_numpy(alpha).cuda()
    ws = plan.alloc_workspace(1)
    g = torch.Generator(device="cuda")
    g.manual_seed(1)
    outs = []
    for fill in ("random", "ones", "stale", "stale"):
        if fill == "random":
            ws.copy_(torch.randint(0, 256, ws.shape, generator=g, device="cuda", dtype=torch.int32).to(torch.uint8))
        elif fill == "ones":
            ws.fill_(0xFF)
        outs.append(plan.forward(tiled, al, x, ws=ws).cpu().numpy())
        assert sdq.sdq_workspace_status(plan.handle, 1, ws) == 0
    yr = O.forward_code_domain(W.bf16_to_float(bits), codes, alpha, 128, d.n_b, signs)
    assert _rel(outs[0], yr) <= 1e-3
    for o in outs[1:]:
        assert np.array_equal(o, outs[0])   # same call shape: deterministic, bit for bit


def test_one_workspace_serves_several_layers(sdq, torch_cuda):
    """Layers with different row-tile counts and split-K grids take turns on
    one workspace (sized for the largest), fused and two-kernel calls mixed."""
    torch = torch_cuda
    layers = [_layer(sdq, torch, n, k, 128, 2, O.TERNARY, seed=n) for n, k in
              [(1024, 8192), (4096, 1024), (640, 2048)]]
    ms = [1, 4, 2]
    size = max(sdq.sdq_workspace_bytes(lay[0].handle, m) for lay in layers for m in ms + [8])
    ws = torch.empty(size, dtype=torch.uint8, device="cuda")
    ws.fill_(0x5A)
    for rnd in range(2):
        for i, (plan, d, signs, codes, alpha, tiled) in enumerate(layers):
            m = ms[(i + rnd) % 3] if rnd == 0 else 8   # 8: the two-kernel path
            bits, x = _x(torch, m, d.k_in, seed=17 * i + m)
            y = plan.forward(tiled, torch.from_numpy(alpha).cuda(), x, ws=ws).cpu().numpy()
            assert sdq.sdq_workspace_status(plan.handle, m, ws) == 0
            yr = O.forward_code_domain(W.bf16_to_float(bits), codes, alpha, 128, d.n_b, signs)
            assert _rel(y, yr) <= 1e-3, (rnd, i, m)


@pytest.mark.parametrize("name", ["q", "k", "gate", "down"])
def test_llama70b_decode_is_one_kernel(sdq, torch_cuda, name):
    """The LLaMA-70B layer's linears run their M = 1 decode as one kernel
    (the bench's workload), and not for batches past the fusion bound."""
    torch = torch_cuda
    cfg = W.config(4)
    lin = [l for l in cfg.linears if l.name == name][0]
    d = sdq.LayerDesc(lin.n_out, lin.k_in, cfg.block, Fraction(lin.osr), cfg.quantizer, 1, 0)
    plan = sdq.Plan(d)
    x = torch.zeros((16, lin.k_in), dtype=torch.bfloat16, device="cuda")
    assert sdq.sdq_forward_kernels(plan.handle, 1, x) == 1
    assert sdq.sdq_forward_kernels(plan.handle, 8, x) == 2
    assert sdq.sdq_forward_kernels(plan.handle, 1, x.view(-1)[1:]) == 2   # misaligned x
