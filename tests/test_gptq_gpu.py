"""GPU parity of the encoder with GPTQ block compensation
(sdq_encode_rows_gptq) against the oracle's canonical fp32 definition
(oracle.encode_gptq): codes and alpha bit-exact on the same W and the same
fp32 factor U of the same synthetic calibration Hessian."""
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


def _factor32(k, tokens, seed):
    x = W.calibration_activations(k, tokens, seed)
    return O.gptq_factor(O.gptq_hessian(x)).astype(np.float32)


def _run(sdq, torch, w, u32, block, osr, q, am=0, had=1, signs=None):
    n, k = w.shape
    d = sdq.LayerDesc(n, k, block, Fraction(osr), q, had, am)
    plan = sdq.Plan(d, signs if had else None)
    codes, alpha = plan.encode_gptq(torch.from_numpy(w).cuda(), torch.from_numpy(u32).cuda())
    torch.cuda.synchronize()
    got = codes.cpu().numpy().view(np.uint32).reshape(n, -1)
    return plan, d, got, alpha.cpu().numpy()


CASES = [
    # n, k, B, OSR, quantizer, alpha mode, hadamard
    (72, 512, 128, 2, O.TERNARY, 0, 1),
    (40, 384, 128, Fraction(5, 2), O.BINARY, 0, 1),
    (33, 512, 128, Fraction(17, 16), O.TERNARY, 0, 1),   # blocks end inside a code word
    (64, 256, 128, 3, O.TERNARY, 1, 1),                  # MEANABS alpha
    (24, 1024, 512, 2, O.TERNARY, 0, 1),                 # B = 512
    (50, 384, 64, Fraction(9, 4), O.BINARY, 0, 0),       # no Hadamard, B = 64
    (130, 640, 128, Fraction(3, 2), O.TERNARY, 0, 1),    # more than one row tile of the update
]


@pytest.mark.parametrize("n,k,block,osr,q,am,had", CASES)
def test_gptq_encode_bit_exact(sdq, torch_cuda, n, k, block, osr, q, am, had):
    rng = np.random.default_rng(n * 1000 + k)
    w = W.weights(W.Linear("g", n, k, Fraction(osr), "t5", 0.02, 77 + n))
    signs = np.where(rng.random(block) < 0.5, -1, 1).astype(np.int8)
    u32 = _factor32(k, 2 * k, n + k)
    _, d, got, alpha = _run(sdq, torch_cuda, w, u32, block, osr, q, am, had, signs)
    oc, oa = O.encode_gptq(w, u32, block, d.n_b, q, am, signs if had else None, bool(had))
    assert np.array_equal(alpha, oa), "alpha differs"
    want = O.pack_plain(oc, q)
    mism = np.mean(got != want)
    assert mism == 0.0, f"code word mismatch rate {mism}"
    # compensation is active: the codes differ from the uncompensated encoder's
    pc, _ = O.encode(w, block, d.n_b, q, am, signs if had else None, bool(had))
    assert not np.array_equal(oc, pc)


def test_gptq_diagonal_factor_matches_plain_encoder(sdq, torch_cuda):
    n, k, block = 48, 512, 128
    w = W.weights(W.Linear("g", n, k, Fraction(2), "normal", 0.02, 5))
    u32 = np.diag(np.full(k, 0.5, dtype=np.float32))
    plan, d, got, alpha = _run(sdq, torch_cuda, w, u32, block, 2, O.TERNARY, signs=None, had=0)
    codes, a2 = plan.encode(torch_cuda.from_numpy(w).cuda())
    assert np.array_equal(got, codes.cpu().numpy().view(np.uint32).reshape(n, -1))
    assert np.array_equal(alpha, a2.cpu().numpy())


def test_gptq_full_size_sampled_rows(sdq, torch_cuda):
    """LLaMA-7B q projection (4096 x 4096, OSR 2, B = 128): every row on the
    GPU, 8 sampled rows through the oracle (rows are independent under the
    compensation: each row's update uses only its own error)."""
    cfg = W.config(2)
    lin = cfg.linears[0]
    w = W.weights(lin)
    signs = W.hadamard_signs(lin, cfg.block)
    u32 = _factor32(lin.k_in, lin.k_in, 2024)
    _, d, got, alpha = _run(sdq, torch_cuda, w, u32, cfg.block, lin.osr, cfg.quantizer, signs=signs)
    rows = np.random.default_rng(9).choice(lin.n_out, 8, replace=False)
    oc, oa = O.encode_gptq(w[rows], u32, cfg.block, d.n_b, cfg.quantizer, signs=signs)
    assert np.array_equal(alpha[rows], oa)
    assert np.array_equal(got[rows], O.pack_plain(oc, cfg.quantizer))


def test_gptq_bad_arguments(sdq, torch_cuda):
    import ctypes
    torch = torch_cuda
    d = sdq.LayerDesc(16, 256, 128, Fraction(2), O.TERNARY, 1, 0)
    plan = sdq.Plan(d)
    w = torch.zeros((16, 256), device="cuda")
    u = torch.eye(256, device="cuda")
    codes = plan.alloc_plain()
    alpha = torch.empty(16, device="cuda")
    need = sdq.sdq_gptq_workspace_bytes(plan.handle)
    assert need >= 16 * 256 * 4 + 16 * 128 * 4
    ws = torch.empty(need, dtype=torch.uint8, device="cuda")
    L = sdq.lib()
    st = L.sdq_encode_rows_gptq(plan.handle, w.data_ptr(), u.data_ptr(), codes.data_ptr(), alpha.data_ptr(),
                                ws.data_ptr(), need - 1, None)
    assert st == -3                                   # SDQ_ERR_WORKSPACE
    st = L.sdq_encode_rows_gptq(plan.handle, w.data_ptr() + 4, u.data_ptr(), codes.data_ptr(),
                                alpha.data_ptr(), ws.data_ptr(), need, None)
    assert st == -1                                   # misaligned W
    st = L.sdq_encode_rows_gptq(plan.handle, None, u.data_ptr(), codes.data_ptr(), alpha.data_ptr(),
                                ws.data_ptr(), need, None)
    assert st == -1
    assert L.sdq_gptq_workspace_bytes(None) == 0
    d2 = sdq.LayerDesc(16, 16, 2, Fraction(2), O.TERNARY, 1, 0)   # B = 2: not a multiple of 4
    p2 = sdq.Plan(d2)
    st = L.sdq_encode_rows_gptq(p2.handle, w.data_ptr(), u.data_ptr(), codes.data_ptr(), alpha.data_ptr(),
                                ws.data_ptr(), need, None)
    assert st == -2                                   # SDQ_ERR_UNSUPPORTED
    del ctypes
