"""Seeded synthetic workloads shaped like the paper's OPT / LLaMA linears.

This module holds no SDQ arithmetic: only shapes, distributions and seeds.
It is the one module that both the oracle-side tests and the CUDA-side
callers use to make inputs, so that both read identical bytes.

The paper evaluates on pretrained OPT / LLaMA checkpoints with WikiText2 / C4
(section 4.1); none of those are available, so synthetic weights with the
same linear shapes stand in for them:

* single-256x512  one 256 x 512 linear, W ~ N(0, 0.02), B = 512, OSR 2, ternary, M = 1.
* opt-125m  OPT-125M decoder linears (q/k/v/o 768x768, fc1 3072x768, fc2
        768x3072), W ~ N(0, 0.02) with round(0.005 K) outlier input columns
        scaled x20, OSR 2.5, binary, M in {1, 16}.
* llama-7b-layer  LLaMA-7B decoder linears (q/k/v/o 4096^2, gate/up 11008x4096, down
        4096x11008), Student-t(5) scaled to std 0.02 times a per-row factor
        log-uniform in [0.5, 2], OSR 2, ternary, M in {1, 4, 16, 64}.
* llama-13b-4layers  LLaMA-13B 4-layer stack (q/k/v/o 5120^2, gate/up 13824x5120, down
        5120x13824), N(0, sigma_l) with sigma_l log-uniform in [0.01, 0.03]
        per linear, MultiOSR in {1.5, 2, 2.5, 3}, ternary, M = 8 and 2048.
* llama-70b-layer  LLaMA-70B decoder layer (q/o 8192^2, k/v 1024x8192, gate/up
        28672x8192, down 8192x28672), Student-t(5) scaled to std 0.015,
        OSR 2, ternary, M = 4096 (prefill) and 1..64 (decode).

Activations: x ~ N(0, 1) rounded to bf16.  GPTQ calibration activations:
:func:`calibration_activations` (correlated channels with outliers).  Hadamard sign vectors: +-1 drawn
uniformly.  Seeds: ``20251003 + 1000 * index + linear`` (weights; activations
``+ 250``; Hadamard signs ``+ 500``).  Matrices are (N, K) = (out, in).
"""
from __future__ import annotations

from dataclasses import dataclass, field
from fractions import Fraction

import numpy as np

BASE_SEED = 20251003
TERNARY = 2
BINARY = 1


@dataclass(frozen=True)
class Linear:
    name: str
    n_out: int
    k_in: int
    osr: Fraction
    dist: str                 # "normal", "normal_outliers", "t5_rowscale", "t5"
    std: float
    seed: int


@dataclass
class Config:
    index: int
    name: str
    block: int
    quantizer: int
    linears: list = field(default_factory=list)
    decode_batches: tuple = (1,)
    prefill_batch: int = 0

    def n_b(self, lin: Linear) -> int:
        nb = self.block * lin.osr
        assert nb.denominator == 1, "OSR * B must be an integer"
        return int(nb)


def _seed(cfg: int, lin: int) -> int:
    return BASE_SEED + 1000 * cfg + lin


def _llama_layer(cfg, hidden, ffn, kv, osr, dist, std, layer=0, prefix=""):
    shapes = [("q", hidden, hidden), ("k", kv, hidden), ("v", kv, hidden),
              ("o", hidden, hidden), ("gate", ffn, hidden), ("up", ffn, hidden),
              ("down", hidden, ffn)]
    out = []
    for i, (nm, n, k) in enumerate(shapes):
        li = 7 * layer + i
        o = osr[i] if isinstance(osr, (list, tuple)) else osr
        s = std[i] if isinstance(std, (list, tuple)) else std
        out.append(Linear(prefix + nm, n, k, Fraction(o), dist, s, _seed(cfg, li)))
    return out


def config(index: int, multiosr=None) -> Config:
    """The synthetic workload ``index`` (0..4).  For llama-13b-4layers the per-linear OSR
    map comes from ``multiosr`` (a callable taking the list of (params,
    variance) per layer, see ``paper_2510_03275_gb300.multiosr``); without it
    every llama-13b-4layers linear uses OSR 2."""
    if index == 0:
        c = Config(0, "single-256x512", 512, TERNARY, decode_batches=(1,))
        c.linears = [Linear("lin", 256, 512, Fraction(2), "normal", 0.02, _seed(0, 0))]
        return c
    if index == 1:
        c = Config(1, "opt-125m", 128, BINARY, decode_batches=(1, 16))
        shapes = [("q", 768, 768), ("k", 768, 768), ("v", 768, 768), ("o", 768, 768),
                  ("fc1", 3072, 768), ("fc2", 768, 3072)]
        c.linears = [Linear(nm, n, k, Fraction(5, 2), "normal_outliers", 0.02, _seed(1, i))
                     for i, (nm, n, k) in enumerate(shapes)]
        return c
    if index == 2:
        c = Config(2, "llama-7b-layer", 128, TERNARY, decode_batches=(1, 4, 16, 64))
        c.linears = _llama_layer(2, 4096, 11008, 4096, 2, "t5_rowscale", 0.02)
        return c
    if index == 3:
        c = Config(3, "llama-13b-4layers", 128, TERNARY, decode_batches=(8,),
                   prefill_batch=2048)
        rng = np.random.default_rng(_seed(3, 999))
        stds = np.exp(rng.uniform(np.log(0.01), np.log(0.03), size=(4, 7)))
        osrs = [[2] * 7 for _ in range(4)]
        if multiosr is not None:
            sizes = [[n * k for _, n, k in _13b_shapes()] for _ in range(4)]
            osrs = multiosr(sizes, (stds ** 2).tolist())
        lins = []
        for layer in range(4):
            lins += _llama_layer(3, 5120, 13824, 5120, [Fraction(o) for o in osrs[layer]],
                                 "normal", stds[layer].tolist(), layer, f"l{layer}.")
        c.linears = lins
        return c
    if index == 4:
        c = Config(4, "llama-70b-layer", 128, TERNARY,
                   decode_batches=(1, 2, 4, 8, 16, 32, 64), prefill_batch=4096)
        c.linears = _llama_layer(4, 8192, 28672, 1024, 2, "t5", 0.015)
        return c
    raise ValueError("config index must be 0..4")


def shared_input_groups(cfg: Config):
    """The linears of ``cfg`` that read the same input, as (name, [Linear])
    groups in layer order: q/k/v (attention input) and gate/up (MLP input)
    of each decoder layer when their OSRs agree; every other linear alone.
    One plan over the rows of a group (rows concatenated, one Hadamard sign
    vector) computes every member's output: alpha and codes are per row."""
    groups, i, lins = [], 0, cfg.linears
    while i < len(lins):
        pre, base = lins[i].name.rpartition(".")[0], lins[i].name.rpartition(".")[2]
        members = [lins[i]]
        want = {"q": ("k", "v"), "gate": ("up",)}.get(base, ())
        for j, nm in enumerate(want, 1):
            if i + j < len(lins) and lins[i + j].name == (pre + "." if pre else "") + nm \
                    and lins[i + j].osr == lins[i].osr and lins[i + j].k_in == lins[i].k_in:
                members.append(lins[i + j])
            else:
                break
        if len(members) != 1 + len(want):
            members = [lins[i]]
        name = (pre + "." if pre else "") + "_".join(m.name.rpartition(".")[2] for m in members)
        if len(members) == 3:
            name = (pre + "." if pre else "") + "qkv"
        groups.append((name, members))
        i += len(members)
    return groups


def _13b_shapes():
    return [("q", 5120, 5120), ("k", 5120, 5120), ("v", 5120, 5120), ("o", 5120, 5120),
            ("gate", 13824, 5120), ("up", 13824, 5120), ("down", 5120, 13824)]


# ------------------------------------------------------------------ host side
def weights(lin: Linear, rows=None) -> np.ndarray:
    """fp32 weights (n_out, k_in) of ``lin`` from numpy's PCG64; ``rows``
    selects a subset of rows of the same matrix (the full matrix is drawn
    row-block by row-block so any subset is reproducible cheaply)."""
    rows = np.arange(lin.n_out) if rows is None else np.asarray(rows)
    out = np.empty((len(rows), lin.k_in), dtype=np.float32)
    rb = 256                                   # rows drawn per sub-stream
    blocks = np.unique(rows // rb)
    for b in blocks:
        blk = _weight_rowblock(lin, int(b), rb)
        sel = np.nonzero(rows // rb == b)[0]
        out[sel] = blk[rows[sel] - b * rb]
    return out


def _weight_rowblock(lin: Linear, b: int, rb: int) -> np.ndarray:
    n = min(rb, lin.n_out - b * rb)
    rng = np.random.default_rng([lin.seed, b])
    k = lin.k_in
    if lin.dist in ("normal", "normal_outliers"):
        w = rng.standard_normal((n, k)) * lin.std
        if lin.dist == "normal_outliers":
            cols = outlier_columns(lin)
            w[:, cols] *= 20.0
    elif lin.dist in ("t5", "t5_rowscale"):
        w = rng.standard_t(5, (n, k)) * (lin.std / np.sqrt(5.0 / 3.0))
        if lin.dist == "t5_rowscale":
            rs = np.random.default_rng([lin.seed, 7777]).uniform(
                np.log(0.5), np.log(2.0), size=lin.n_out)
            w *= np.exp(rs[b * rb:b * rb + n])[:, None]
    else:
        raise ValueError(lin.dist)
    return w.astype(np.float32)


def outlier_columns(lin: Linear) -> np.ndarray:
    """The round(0.005 K) input columns scaled x20 in opt-125m."""
    cnt = int(round(0.005 * lin.k_in))
    return np.sort(np.random.default_rng([lin.seed, 4242]).permutation(lin.k_in)[:cnt])


def hadamard_signs(lin: Linear, block: int) -> np.ndarray:
    """The random sign vector d (+-1, int8) of the randomised Hadamard."""
    rng = np.random.default_rng(lin.seed + 500)
    return np.where(rng.integers(0, 2, size=block) == 1, 1, -1).astype(np.int8)


def activations(lin: Linear, m: int, seed_offset: int = 250) -> np.ndarray:
    """x ~ N(0, 1) rounded to bf16, returned as the bf16 bit patterns
    (uint16, (m, k_in)); ``bf16_to_float`` gives the values."""
    rng = np.random.default_rng(lin.seed + seed_offset + 7919 * m)
    x = rng.standard_normal((m, lin.k_in)).astype(np.float32)
    return float_to_bf16(x)


def calibration_activations(k_in: int, n_tokens: int, seed: int) -> np.ndarray:
    """Synthetic calibration activations (n_tokens, k_in) fp32 for the GPTQ
    Hessian: channels correlated through a rank-16 shared component, per-
    channel scales log-normal (sigma 0.5) and round(0.005 k_in) outlier
    channels scaled x20 (the outlier-channel structure of LLM activations;
    the paper calibrates on C4 samples, which are not available)."""
    rng = np.random.default_rng([seed, 31337])
    z = rng.standard_normal((n_tokens, k_in))
    f = rng.standard_normal((n_tokens, 16))
    a = rng.standard_normal((16, k_in)) / 4.0
    scale = np.exp(rng.normal(0.0, 0.5, size=k_in))
    scale[rng.permutation(k_in)[:int(round(0.005 * k_in))]] *= 20.0
    return ((z + 2.0 * (f @ a)) * scale).astype(np.float32)


def float_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even fp32 -> bf16 bit patterns (uint16)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)
    return r


def bf16_to_float(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def random_codes(n: int, k: int, quantizer: int, seed: int, p_zero: float = 0.5) -> np.ndarray:
    """Seeded random codes (int8) for contraction-only checks."""
    rng = np.random.default_rng(seed)
    if quantizer == BINARY:
        return np.where(rng.random((n, k)) < 0.5, 1, -1).astype(np.int8)
    u = rng.random((n, k))
    return np.where(u < p_zero, 0, np.where(u < (1 + p_zero) / 2, 1, -1)).astype(np.int8)


# ---------------------------------------------------------------- device side
def weights_device(lin: Linear, device="cuda"):
    """fp32 weights of ``lin`` drawn on the device with torch's Philox
    generator: same distribution as :func:`weights`, different draws.  Used
    where host generation of multi-GB matrices would dominate run time;
    callers that compare against the oracle copy the rows they sample."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(lin.seed)
    n, k = lin.n_out, lin.k_in
    if lin.dist in ("normal", "normal_outliers"):
        w = torch.randn((n, k), generator=g, device=device, dtype=torch.float32) * lin.std
        if lin.dist == "normal_outliers":
            cols = torch.as_tensor(outlier_columns(lin), device=device)
            w[:, cols] *= 20.0
        return w
    # Student-t(5) = Z / sqrt(V / 5) with V ~ chi^2_5 = 2 * Gamma(5/2).
    z = torch.randn((n, k), generator=g, device=device, dtype=torch.float32)
    gam = torch._standard_gamma(torch.full((n, k), 2.5, device=device), generator=g)
    w = z / torch.sqrt(gam * (2.0 / 5.0)) * (lin.std / float(np.sqrt(5.0 / 3.0)))
    if lin.dist == "t5_rowscale":
        rs = np.random.default_rng([lin.seed, 7777]).uniform(np.log(0.5), np.log(2.0), size=n)
        w *= torch.as_tensor(np.exp(rs), device=device, dtype=torch.float32)[:, None]
    return w
