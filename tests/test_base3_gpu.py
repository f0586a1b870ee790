"""GPU parity of the base-3 storage kernels (sdq_pack_base3 /
sdq_unpack_base3) with the oracle's definition: bytes and plain words
bit-exact, round trips through the tiled layout, and invalid bytes counted."""
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


def _plan(sdq, n, k, osr):
    return sdq.Plan(sdq.LayerDesc(n, k, 128, Fraction(osr), O.TERNARY, 1, 0))


@pytest.mark.parametrize("n,k,osr", [(37, 256, 2), (5, 128, Fraction(17, 16)), (64, 640, Fraction(5, 2)),
                                     (130, 384, 3), (3, 128, 1)])
def test_pack_unpack_base3_bit_exact(sdq, torch_cuda, n, k, osr):
    torch = torch_cuda
    plan = _plan(sdq, n, k, osr)
    d = plan.desc
    k_eff = sdq.sdq_k_eff(d)
    codes = W.random_codes(n, k_eff, O.TERNARY, n + k)
    plain = torch.from_numpy(O.pack_plain(codes, O.TERNARY).reshape(-1).view(np.int32)).cuda()
    nbytes = sdq.sdq_base3_bytes(d)
    assert nbytes == n * O.base3_bytes_per_row(k_eff)
    b3 = torch.full((nbytes,), 0x5A, dtype=torch.uint8, device="cuda")
    sdq.sdq_pack_base3(plan.handle, plain, b3)
    torch.cuda.synchronize()
    want = O.pack_base3(codes)
    assert np.array_equal(b3.cpu().numpy().reshape(n, -1), want)
    back = torch.full_like(plain, -1)
    bad = torch.zeros(1, dtype=torch.int32, device="cuda")
    sdq.sdq_unpack_base3(plan.handle, b3, back, bad)
    torch.cuda.synchronize()
    assert int(bad.item()) == 0
    assert np.array_equal(back.cpu().numpy().view(np.uint32), O.pack_plain(codes, O.TERNARY).reshape(-1))


def test_unpack_base3_counts_invalid_bytes(sdq, torch_cuda):
    torch = torch_cuda
    n, k = 4, 128
    plan = _plan(sdq, n, k, 2)
    k_eff = sdq.sdq_k_eff(plan.desc)
    codes = W.random_codes(n, k_eff, O.TERNARY, 3)
    data = O.pack_base3(codes)
    data[1, 7] = 243
    data[2, 0] = 255
    data[3, 50] = 250
    want, nbad = O.unpack_base3(data, k_eff)
    assert nbad == 3
    plain = torch.empty(sdq.sdq_plain_bytes(plan.desc) // 4, dtype=torch.int32, device="cuda")
    bad = torch.zeros(1, dtype=torch.int32, device="cuda")
    sdq.sdq_unpack_base3(plan.handle, torch.from_numpy(data.reshape(-1)).cuda(), plain, bad)
    torch.cuda.synchronize()
    assert int(bad.item()) == 3
    assert np.array_equal(plain.cpu().numpy().view(np.uint32), O.pack_plain(want, O.TERNARY).reshape(-1))


def test_base3_full_size_layer_round_trip_through_tiled(sdq, torch_cuda):
    """LLaMA-70B gate (28672 x 8192, OSR 2): plain -> base-3 -> plain ->
    tiled equals plain -> tiled, on device-drawn codes; sampled rows of the
    base-3 bytes against the oracle."""
    torch = torch_cuda
    cfg = W.config(4)
    lin = cfg.linears[4]
    plan = _plan(sdq, lin.n_out, lin.k_in, lin.osr)
    d = plan.desc
    k_eff = sdq.sdq_k_eff(d)
    g = torch.Generator(device="cuda")
    g.manual_seed(11)
    plain = torch.randint(-2 ** 31, 2 ** 31 - 1, (sdq.sdq_plain_bytes(d) // 4,), generator=g,
                          dtype=torch.int32, device="cuda")
    # make every field valid (10 -> 00) and the row padding 0: unpack(pack(.)) does that
    tiled0 = plan.alloc_tiled()
    sdq.sdq_pack(plan.handle, plain, tiled0)
    sdq.sdq_unpack(plan.handle, tiled0, plain, None)
    sdq.sdq_pack(plan.handle, plain, tiled0)
    b3 = torch.empty(sdq.sdq_base3_bytes(d), dtype=torch.uint8, device="cuda")
    sdq.sdq_pack_base3(plan.handle, plain, b3)
    back = torch.empty_like(plain)
    sdq.sdq_unpack_base3(plan.handle, b3, back, None)
    tiled1 = plan.alloc_tiled()
    sdq.sdq_pack(plan.handle, back, tiled1)
    torch.cuda.synchronize()
    assert torch.equal(back, plain)
    assert torch.equal(tiled1, tiled0)
    rows = np.random.default_rng(4).choice(lin.n_out, 16, replace=False)
    wpr = O.plain_words_per_row(k_eff, O.TERNARY)
    pl = plain.view(lin.n_out, wpr)[torch.as_tensor(rows, device="cuda")].cpu().numpy().view(np.uint32)
    codes = O.unpack_plain(pl, O.TERNARY, k_eff)
    got = b3.view(lin.n_out, -1)[torch.as_tensor(rows, device="cuda")].cpu().numpy()
    assert np.array_equal(got, O.pack_base3(codes))
    assert b3.numel() / plain.numel() / 4 < 0.81


def test_base3_refuses_binary_and_bad_pointers(sdq, torch_cuda):
    torch = torch_cuda
    pb = sdq.Plan(sdq.LayerDesc(8, 128, 128, Fraction(2), O.BINARY, 1, 0))
    buf = torch.zeros(4096, dtype=torch.int32, device="cuda")
    L = sdq.lib()
    assert L.sdq_pack_base3(pb.handle, buf.data_ptr(), buf.data_ptr() + 8192, None) == -2
    pt = _plan(sdq, 8, 128, 2)
    assert L.sdq_pack_base3(pt.handle, buf.data_ptr() + 4, buf.data_ptr() + 8192, None) == -1
    assert L.sdq_unpack_base3(pt.handle, None, buf.data_ptr(), None, None) == -1
