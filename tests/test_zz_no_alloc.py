"""The allocation-free decode entry point against the workspace one.

sdq_linear_forward_noalloc serves callers that may not allocate device
memory themselves (for instance a plugin whose host runtime owns all device
allocations, or a serving loop that forbids allocation after start-up): it
runs the same kernels on a library-owned device array.  This file is
collected last so that a failure here does not hide the other GPU tests.
"""
from fractions import Fraction

import numpy as np
import pytest

import oracle as O
from paper_2510_03275_gb300 import workloads as W

pytestmark = pytest.mark.gpu

TOL = 1e-2


def _layer(sdq, torch, n, k, b, osr, q, seed):
    d = sdq.LayerDesc(n, k, b, Fraction(osr), q)
    plan = sdq.Plan(d)
    keff = sdq.sdq_k_eff(d)
    codes = W.random_codes(n, keff, q, seed)
    plain = torch.from_numpy(O.pack_plain(codes, q).ravel().view(np.int32)).cuda()
    tiled = plan.pack(plain)
    alpha = torch.from_numpy((np.random.default_rng(seed).random(n) * 0.05 + 0.01).astype(np.float32)).cuda()
    return plan, tiled, alpha


@pytest.mark.parametrize("shape,m", [((300, 384, 128, Fraction(5, 2), 2), 1),
                                     ((1024, 2048, 128, 2, 2), 4),
                                     ((256, 512, 512, 2, 1), 16)])
def test_noalloc_matches_workspace_forward_twice(sdq, shape, m):
    import torch
    assert torch.cuda.is_available()
    n, k, b, osr, q = shape
    plan, tiled, alpha = _layer(sdq, torch, n, k, b, osr, q, seed=n + m)
    ws = plan.alloc_workspace(m)
    for call in range(2):
        x = torch.randn(m, k, device="cuda").to(torch.bfloat16)
        y_ref = torch.empty((m, n), device="cuda")
        sdq.sdq_linear_forward(plan.handle, tiled, alpha, x, m, y_ref, ws)
        y = torch.full((m, n), float("nan"), device="cuda")
        sdq.sdq_linear_forward_noalloc(plan.handle, tiled, alpha, x, m, y)
        torch.cuda.synchronize()
        a, r = y.cpu().numpy(), y_ref.cpu().numpy()
        assert np.isfinite(a).all(), f"call {call}"
        err = np.abs(a - r).max() / np.abs(r).max()
        assert err <= TOL, (call, err)


def test_noalloc_rejects_oversize(sdq):
    """A workspace need above the fixed array is refused before any launch."""
    import torch
    d = sdq.LayerDesc(8192, 28672, 128, Fraction(2), 2)
    plan = sdq.Plan(d)
    assert sdq.sdq_workspace_bytes(plan.handle, 64) > sdq.sdq_noalloc_scratch_bytes()
    x = torch.zeros((64, 28672), dtype=torch.bfloat16, device="cuda")
    y = torch.zeros((64, 8192), device="cuda")
    tiled = torch.zeros(sdq.sdq_tiled_bytes(d) // 4, dtype=torch.int32, device="cuda")
    alpha = torch.ones(8192, device="cuda")
    with pytest.raises(sdq.SdqError) as e:
        sdq.sdq_linear_forward_noalloc(plan.handle, tiled, alpha, x, 64, y)
    assert e.value.status == -3
    with pytest.raises(sdq.SdqError) as e:
        sdq.sdq_linear_forward_noalloc(plan.handle, tiled, alpha, x, 65, y)
    assert e.value.status == -1
