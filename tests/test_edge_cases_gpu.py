"""GPU: degenerate and extreme inputs of the forward against the oracle —
zero activations and zero codes, activations scaled by 2^+-100, a single
output row, the smallest and largest Hadamard blocks (B = 2, n_b = 4096),
and invalid batch sizes."""
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


def _layer(sdq, torch, n, k, b, osr, q, seed, zero_codes=False):
    d = sdq.LayerDesc(n, k, b, Fraction(osr), q, 1, 0)
    rng = np.random.default_rng(seed)
    signs = np.where(rng.random(b) < 0.5, -1, 1).astype(np.int8)
    plan = sdq.Plan(d, signs)
    keff = sdq.sdq_k_eff(d)
    codes = W.random_codes(n, keff, q, seed)
    if zero_codes:
        codes = np.zeros_like(codes)
    plain = torch.from_numpy(O.pack_plain(codes, q).ravel().view(np.int32)).cuda()
    tiled = plan.pack(plain)
    alpha = (rng.random(n) * 0.05 + 0.01).astype(np.float32)
    return plan, d, signs, codes, alpha, tiled


def _forward(sdq, torch, lay, xf):
    plan, d, signs, codes, alpha, tiled = lay
    bits = W.float_to_bf16(xf.astype(np.float32))
    x = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).cuda()
    ws = plan.alloc_workspace(x.shape[0])
    y = plan.forward(tiled, torch.from_numpy(alpha).cuda(), x, ws=ws).cpu().numpy()
    assert sdq.sdq_workspace_status(plan.handle, x.shape[0], ws) == 0
    yr = O.forward_code_domain(W.bf16_to_float(bits), codes, alpha, d.block, d.n_b, signs)
    return y, yr


@pytest.mark.parametrize("m", [1, 3, 12, 70])
def test_zero_activations_and_zero_codes(sdq, torch_cuda, m):
    torch = torch_cuda
    lay = _layer(sdq, torch, 200, 1024, 128, 2, O.TERNARY, seed=m)
    y, _ = _forward(sdq, torch, lay, np.zeros((m, 1024)))
    assert np.all(y == 0.0)
    lay0 = _layer(sdq, torch, 200, 1024, 128, 2, O.TERNARY, seed=m, zero_codes=True)
    y, _ = _forward(sdq, torch, lay0, np.random.default_rng(m).standard_normal((m, 1024)))
    assert np.all(y == 0.0)


@pytest.mark.parametrize("m", [1, 4, 9, 70])
@pytest.mark.parametrize("scale", [2.0 ** 100, 2.0 ** -100])
def test_extreme_activation_scales(sdq, torch_cuda, m, scale):
    """The per-row power-of-two term scale makes the result scale-invariant."""
    torch = torch_cuda
    lay = _layer(sdq, torch, 300, 2048, 128, 2, O.TERNARY, seed=5 + m)
    xf = np.random.default_rng(m).standard_normal((m, 2048)) * scale
    y, yr = _forward(sdq, torch, lay, xf)
    assert np.all(np.isfinite(y))
    err = np.abs(y - yr).max() / np.abs(yr).max()
    assert err <= (1e-3 if m <= 8 else 8e-3), err


@pytest.mark.parametrize("q", [O.TERNARY, O.BINARY])
@pytest.mark.parametrize("n,k,b,osr,m", [(1, 16, 16, 1, 1), (1, 256, 128, Fraction(5, 2), 2),
                                         (3, 8, 2, Fraction(3, 2), 1), (5, 64, 2, 2, 66),
                                         (40, 2048, 1024, 4, 1), (40, 2048, 1024, 4, 70)])
def test_degenerate_shapes(sdq, torch_cuda, q, n, k, b, osr, m):
    """One output row; the smallest Hadamard block (B = 2); the largest
    upsampled block (B = 1024 at OSR 4: n_b = 4096)."""
    torch = torch_cuda
    lay = _layer(sdq, torch, n, k, b, osr, q, seed=n * 31 + k + m)
    y, yr = _forward(sdq, torch, lay, np.random.default_rng(n + m).standard_normal((m, k)))
    err = np.abs(y - yr).max() / np.abs(yr).max()
    assert err <= 1e-2, err


def test_invalid_batch_rejected(sdq, torch_cuda):
    torch = torch_cuda
    plan, d, signs, codes, alpha, tiled = _layer(sdq, torch, 64, 256, 128, 2, O.TERNARY, seed=1)
    x = torch.zeros((1, 256), dtype=torch.bfloat16, device="cuda")
    y = torch.empty((1, 64), device="cuda")
    ws = plan.alloc_workspace(1)
    al = torch.from_numpy(alpha).cuda()
    for bad_m in (0, -1, 65536):
        with pytest.raises(sdq.SdqError) as e:
            sdq.sdq_linear_forward(plan.handle, tiled, al, x, bad_m, y, ws)
        assert e.value.status == -1
    assert sdq.sdq_forward_kernels(plan.handle, 0, x) == 0
