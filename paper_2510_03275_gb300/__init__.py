"""Python binding of libsdq, the GB300 Sigma-Delta-quantized linear layer.

Thin ctypes layer over the C ABI in ``include/sdq.h``: the functions below
carry the C names and only marshal arguments (pointers, sizes, streams).  All
compute runs in the CUDA kernels of ``libsdq.so``; there is no CPU path.  If
the library is missing, every call raises ``RuntimeError`` -- build it with
``python -m paper_2510_03275_gb300.build``.

Tensors are PyTorch tensors (device memory and streams only).  bf16
activations are passed as ``torch.bfloat16`` tensors; codes as ``torch.int32``
tensors holding the uint32 words.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from fractions import Fraction

__all__ = [
    "SDQ_OK", "SDQ_BINARY", "SDQ_TERNARY", "SDQ_ALPHA_MAXABS", "SDQ_ALPHA_MEANABS",
    "SdqError", "LayerDesc", "lib", "library_path",
    "sdq_plan_create", "sdq_plan_destroy", "sdq_k_eff", "sdq_plain_bytes", "sdq_tiled_bytes",
    "sdq_workspace_bytes", "sdq_build_tables", "sdq_build_gptq_table", "sdq_decode_launch_shape", "sdq_encode_rows", "sdq_gptq_workspace_bytes",
    "sdq_encode_rows_gptq", "sdq_base3_bytes", "sdq_pack_base3", "sdq_unpack_base3", "sdq_pack", "sdq_unpack",
    "sdq_prep_activations", "sdq_contract", "sdq_contract_add", "sdq_linear_forward", "sdq_read_prep",
    "sdq_workspace_status", "sdq_linear_forward_noalloc", "sdq_noalloc_scratch_bytes", "sdq_noalloc_status",
    "sdq_forward_kernels", "sdq_forward_route", "sdq_status_string", "Plan",
]

SDQ_OK = 0
SDQ_BINARY = 1
SDQ_TERNARY = 2
SDQ_ALPHA_MAXABS = 0
SDQ_ALPHA_MEANABS = 1

_HERE = os.path.dirname(os.path.abspath(__file__))
library_path = os.path.join(_HERE, "libsdq.so")


class SdqError(RuntimeError):
    def __init__(self, status: int, where: str):
        msg = lib().sdq_status_string(status).decode() if _lib is not None else str(status)
        super().__init__(f"{where}: {msg}")
        self.status = status


class _Desc(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("n_out", "k_in", "block", "osr_num", "osr_den", "quantizer", "hadamard",
                 "alpha_mode")]


@dataclass(frozen=True)
class LayerDesc:
    """Mirror of ``sdq_layer_desc``: OSR is a Fraction (num/den)."""
    n_out: int
    k_in: int
    block: int
    osr: Fraction
    quantizer: int = SDQ_TERNARY
    hadamard: int = 1
    alpha_mode: int = SDQ_ALPHA_MAXABS

    def c(self) -> _Desc:
        o = Fraction(self.osr)
        return _Desc(self.n_out, self.k_in, self.block, o.numerator, o.denominator,
                     self.quantizer, self.hadamard, self.alpha_mode)

    @property
    def n_b(self) -> int:
        return int(self.block * Fraction(self.osr))


_lib = None
_vp, _sz, _i32, _i64 = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int32, ctypes.c_int64
_SIGS = {
    "sdq_plan_create": (ctypes.c_int, [ctypes.POINTER(_Desc), _vp, ctypes.POINTER(_vp)]),
    "sdq_plan_destroy": (ctypes.c_int, [_vp]),
    "sdq_k_eff": (_i64, [ctypes.POINTER(_Desc)]),
    "sdq_plain_bytes": (_sz, [ctypes.POINTER(_Desc)]),
    "sdq_tiled_bytes": (_sz, [ctypes.POINTER(_Desc)]),
    "sdq_workspace_bytes": (_sz, [_vp, _i32]),
    "sdq_build_tables": (ctypes.c_int, [ctypes.POINTER(_Desc), _vp, _vp, _vp]),
    "sdq_build_gptq_table": (ctypes.c_int, [ctypes.POINTER(_Desc), _vp, _vp]),
    "sdq_decode_launch_shape": (ctypes.c_int, [ctypes.POINTER(_Desc), _i32, _i32, _vp]),
    "sdq_encode_rows": (ctypes.c_int, [_vp, _vp, _vp, _vp, _vp]),
    "sdq_gptq_workspace_bytes": (ctypes.c_size_t, [_vp]),
    "sdq_base3_bytes": (ctypes.c_size_t, [ctypes.POINTER(_Desc)]),
    "sdq_pack_base3": (ctypes.c_int, [_vp, _vp, _vp, _vp]),
    "sdq_unpack_base3": (ctypes.c_int, [_vp, _vp, _vp, _vp, _vp]),
    "sdq_encode_rows_gptq": (ctypes.c_int, [_vp, _vp, _vp, _vp, _vp, _vp, ctypes.c_size_t, _vp]),
    "sdq_pack": (ctypes.c_int, [_vp, _vp, _vp, _vp]),
    "sdq_unpack": (ctypes.c_int, [_vp, _vp, _vp, _vp, _vp]),
    "sdq_prep_activations": (ctypes.c_int, [_vp, _vp, _i32, _vp, _sz, _vp]),
    "sdq_contract": (ctypes.c_int, [_vp, _vp, _vp, _i32, _vp, _vp, _sz, _vp]),
    "sdq_contract_add": (ctypes.c_int, [_vp, _vp, _vp, _i32, _vp, _vp, _sz, _vp]),
    "sdq_linear_forward": (ctypes.c_int, [_vp, _vp, _vp, _vp, _i32, _vp, _vp, _sz, _vp]),
    "sdq_read_prep": (ctypes.c_int, [_vp, _i32, _vp, _vp, _vp]),
    "sdq_workspace_status": (ctypes.c_int, [_vp, _i32, _vp, _vp]),
    "sdq_forward_kernels": (ctypes.c_int, [_vp, _i32, _vp]),
    "sdq_forward_route": (ctypes.c_int, [_vp, _i32]),
    "sdq_linear_forward_noalloc": (ctypes.c_int, [_vp, _vp, _vp, _vp, _i32, _vp, _vp]),
    "sdq_noalloc_status": (ctypes.c_int, [_vp, _i32, _vp]),
    "sdq_noalloc_scratch_bytes": (_sz, []),
    "sdq_status_string": (ctypes.c_char_p, [ctypes.c_int]),
}


def lib():
    """Load libsdq.so (once); raise if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(library_path):
            raise RuntimeError(f"libsdq.so not found at {library_path}; run "
                               "`python -m paper_2510_03275_gb300.build` (CUDA toolkit needed)")
        L = ctypes.CDLL(library_path)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype, f.argtypes = res, args
        _lib = L
    return _lib


def _check(st: int, where: str):
    if st != SDQ_OK:
        raise SdqError(st, where)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


# ------------------------------------------------------------- C-ABI names
def sdq_plan_create(desc: LayerDesc, had_signs=None) -> int:
    import numpy as np
    d = desc.c()
    h = ctypes.c_void_p()
    signs = None
    if had_signs is not None:
        signs = np.ascontiguousarray(had_signs, dtype=np.int8)
    st = lib().sdq_plan_create(ctypes.byref(d),
                               None if signs is None else signs.ctypes.data_as(_vp),
                               ctypes.byref(h))
    _check(st, "sdq_plan_create")
    return h.value


def sdq_plan_destroy(plan: int):
    _check(lib().sdq_plan_destroy(plan), "sdq_plan_destroy")


def sdq_k_eff(desc: LayerDesc) -> int:
    return lib().sdq_k_eff(ctypes.byref(desc.c()))


def sdq_plain_bytes(desc: LayerDesc) -> int:
    return lib().sdq_plain_bytes(ctypes.byref(desc.c()))


def sdq_tiled_bytes(desc: LayerDesc) -> int:
    return lib().sdq_tiled_bytes(ctypes.byref(desc.c()))


def sdq_workspace_bytes(plan: int, M: int) -> int:
    return lib().sdq_workspace_bytes(plan, M)


def sdq_build_tables(desc: LayerDesc, had_signs=None):
    """Host-only: (A_enc, G) as float32 numpy arrays (n_b x B)."""
    import numpy as np
    a = np.zeros((desc.n_b, desc.block), np.float32)
    g = np.zeros((desc.n_b, desc.block), np.float32)
    signs = None if had_signs is None else np.ascontiguousarray(had_signs, dtype=np.int8)
    st = lib().sdq_build_tables(ctypes.byref(desc.c()),
                                None if signs is None else signs.ctypes.data_as(_vp),
                                a.ctypes.data_as(_vp), g.ctypes.data_as(_vp))
    _check(st, "sdq_build_tables")
    return a, g


def sdq_build_gptq_table(desc: LayerDesc, had_signs=None):
    """Host-only: the fp32 G of the GPTQ block reconstruction (n_b x B)."""
    import numpy as np
    g = np.zeros((desc.n_b, desc.block), np.float32)
    signs = None if had_signs is None else np.ascontiguousarray(had_signs, dtype=np.int8)
    st = lib().sdq_build_gptq_table(ctypes.byref(desc.c()), None if signs is None else signs.ctypes.data_as(_vp),
                                    g.ctypes.data_as(_vp))
    _check(st, "sdq_build_gptq_table")
    return g


_SHAPE_KEYS = ("T", "NP", "S", "P", "CB", "ring", "sb", "nbuf", "smem", "slot_bytes", "b_bytes", "ss",
               "smem_limit", "npipe", "ns", "bstream")


def sdq_decode_launch_shape(desc: LayerDesc, M: int, sm_count: int) -> dict:
    """Host-only: the decode launch shape at batch M (include/sdq.h)."""
    import numpy as np
    out = np.zeros(len(_SHAPE_KEYS), np.int64)
    _check(lib().sdq_decode_launch_shape(ctypes.byref(desc.c()), M, sm_count, out.ctypes.data_as(_vp)),
           "sdq_decode_launch_shape")
    return dict(zip(_SHAPE_KEYS, (int(v) for v in out)))


def sdq_encode_rows(plan, W, codes_plain, alpha, stream=None):
    _check(lib().sdq_encode_rows(plan, _ptr(W), _ptr(codes_plain), _ptr(alpha), _stream(stream)),
           "sdq_encode_rows")


def sdq_gptq_workspace_bytes(plan) -> int:
    return int(lib().sdq_gptq_workspace_bytes(plan))


def sdq_encode_rows_gptq(plan, W, U, codes_plain, alpha, ws, stream=None):
    _check(lib().sdq_encode_rows_gptq(plan, _ptr(W), _ptr(U), _ptr(codes_plain), _ptr(alpha), _ptr(ws),
                                      ws.numel() * ws.element_size(), _stream(stream)),
           "sdq_encode_rows_gptq")


def sdq_base3_bytes(desc: LayerDesc) -> int:
    return int(lib().sdq_base3_bytes(ctypes.byref(desc.c())))


def sdq_pack_base3(plan, codes_plain, codes_base3, stream=None):
    _check(lib().sdq_pack_base3(plan, _ptr(codes_plain), _ptr(codes_base3), _stream(stream)), "sdq_pack_base3")


def sdq_unpack_base3(plan, codes_base3, codes_plain, bad_count=None, stream=None):
    _check(lib().sdq_unpack_base3(plan, _ptr(codes_base3), _ptr(codes_plain),
                                  None if bad_count is None else _ptr(bad_count), _stream(stream)),
           "sdq_unpack_base3")


def sdq_pack(plan, codes_plain, codes_tiled, stream=None):
    _check(lib().sdq_pack(plan, _ptr(codes_plain), _ptr(codes_tiled), _stream(stream)), "sdq_pack")


def sdq_unpack(plan, codes_tiled, codes_plain, bad_count=None, stream=None):
    _check(lib().sdq_unpack(plan, _ptr(codes_tiled), _ptr(codes_plain), _ptr(bad_count),
                            _stream(stream)), "sdq_unpack")


def sdq_prep_activations(plan, x, M, ws, stream=None):
    _check(lib().sdq_prep_activations(plan, _ptr(x), M, _ptr(ws), ws.numel() * ws.element_size(),
                                      _stream(stream)), "sdq_prep_activations")


def sdq_contract(plan, codes_tiled, alpha, M, y, ws, stream=None):
    _check(lib().sdq_contract(plan, _ptr(codes_tiled), _ptr(alpha), M, _ptr(y), _ptr(ws),
                              ws.numel() * ws.element_size(), _stream(stream)), "sdq_contract")


def sdq_contract_add(plan, codes_tiled, alpha, M, y, ws, stream=None):
    """y += the contraction (M <= 64; float reductions, order not fixed)."""
    _check(lib().sdq_contract_add(plan, _ptr(codes_tiled), _ptr(alpha), M, _ptr(y), _ptr(ws),
                                  ws.numel() * ws.element_size(), _stream(stream)), "sdq_contract_add")


def sdq_linear_forward(plan, codes_tiled, alpha, x, M, y, ws, stream=None):
    _check(lib().sdq_linear_forward(plan, _ptr(codes_tiled), _ptr(alpha), _ptr(x), M, _ptr(y),
                                    _ptr(ws), ws.numel() * ws.element_size(), _stream(stream)),
           "sdq_linear_forward")


def sdq_read_prep(plan, M, ws, out, stream=None):
    _check(lib().sdq_read_prep(plan, M, _ptr(ws), _ptr(out), _stream(stream)), "sdq_read_prep")


def sdq_workspace_status(plan, M, ws, stream=None) -> int:
    """Synchronize and return the status of the last decode using ``ws``."""
    return lib().sdq_workspace_status(plan, M, _ptr(ws), _stream(stream))


def sdq_forward_kernels(plan, M, x) -> int:
    """Number of kernels sdq_linear_forward launches (2)."""
    return lib().sdq_forward_kernels(plan, M, _ptr(x))


def sdq_forward_route(plan, M) -> int:
    """Route of sdq_linear_forward at batch M: 1 decode, 2 code-domain
    prefill, 3 dense (weights rebuilt, then one GEMM); see include/sdq.h."""
    return lib().sdq_forward_route(plan, M)


def sdq_linear_forward_noalloc(plan, codes_tiled, alpha, x, M, y, stream=None):
    """Decode forward (M <= 64) using the library's own device scratch array
    instead of a caller workspace; see include/sdq.h for its rules."""
    _check(lib().sdq_linear_forward_noalloc(plan, _ptr(codes_tiled), _ptr(alpha), _ptr(x), M,
                                            _ptr(y), _stream(stream)),
           "sdq_linear_forward_noalloc")


def sdq_noalloc_scratch_bytes() -> int:
    return lib().sdq_noalloc_scratch_bytes()


def sdq_noalloc_status(plan, M, stream=None) -> int:
    """Synchronize and return the status of the last allocation-free call
    with this plan and M on the current device (SDQ_OK or a negative status)."""
    return lib().sdq_noalloc_status(plan, M, _stream(stream))


def sdq_status_string(status: int) -> str:
    return lib().sdq_status_string(status).decode()


# ------------------------------------------------------------ convenience
class Plan:
    """Owns an ``sdq_plan`` plus the device buffers of one quantized layer."""

    def __init__(self, desc: LayerDesc, had_signs=None):
        self.desc = desc
        self.handle = sdq_plan_create(desc, had_signs)
        self.k_eff = sdq_k_eff(desc)

    def close(self):
        if self.handle:
            sdq_plan_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def alloc_plain(self, device="cuda"):
        import torch
        return torch.empty(sdq_plain_bytes(self.desc) // 4, dtype=torch.int32, device=device)

    def alloc_tiled(self, device="cuda"):
        import torch
        return torch.empty(sdq_tiled_bytes(self.desc) // 4, dtype=torch.int32, device=device)

    def alloc_workspace(self, M, device="cuda"):
        import torch
        return torch.empty(sdq_workspace_bytes(self.handle, M), dtype=torch.uint8, device=device)

    def encode(self, W, stream=None):
        """W (n_out x k_in fp32, device) -> (plain codes, alpha)."""
        import torch
        codes = self.alloc_plain(W.device)
        alpha = torch.empty(self.desc.n_out, dtype=torch.float32, device=W.device)
        sdq_encode_rows(self.handle, W.contiguous(), codes, alpha, stream)
        return codes, alpha

    def encode_gptq(self, W, U, stream=None):
        """W (n_out x k_in fp32, device), U (k_in x k_in fp32, device, upper,
        U^T U = H^-1) -> (plain codes, alpha) with GPTQ block compensation."""
        import torch
        codes = self.alloc_plain(W.device)
        alpha = torch.empty(self.desc.n_out, dtype=torch.float32, device=W.device)
        ws = torch.empty(sdq_gptq_workspace_bytes(self.handle), dtype=torch.uint8, device=W.device)
        sdq_encode_rows_gptq(self.handle, W.contiguous(), U.contiguous(), codes, alpha, ws, stream)
        return codes, alpha

    def pack(self, plain, stream=None):
        tiled = self.alloc_tiled(plain.device)
        sdq_pack(self.handle, plain, tiled, stream)
        return tiled

    def forward(self, tiled, alpha, x, ws=None, stream=None):
        """x (M x k_in bf16, device) -> y (M x n_out fp32)."""
        import torch
        M = x.shape[0]
        if ws is None:
            ws = self.alloc_workspace(M, x.device)
        y = torch.empty((M, self.desc.n_out), dtype=torch.float32, device=x.device)
        sdq_linear_forward(self.handle, tiled, alpha, x.contiguous(), M, y, ws, stream)
        return y
