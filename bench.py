"""Benchmark of the SDQ linear-layer hot path on GB300.

Workload (N=1): the LLaMA-70B-shaped decoder layer (q/o 8192x8192, k/v
1024x8192, gate/up 28672x8192, down 8192x28672), OSR 2, ternary codes, B =
128, synthetic Student-t(5) weights (std 0.015) and N(0,1) bf16
activations.  One step = the decode forward (prep + contraction) of all
seven linears at batch M (default 1), as 4 calls: the linears that read the
same input (q/k/v, gate/up) are each one plan over their rows (per-row codes
and alpha: every member's outputs are those of its own plan); the same layer
as 7 calls is reported beside it.  Metric: weight-HBM GB/s = packed code
bytes of the layer / step time.  The code matrices (428 MB) are streamed in
turn, so every step reads them from HBM (L2 is 129 MB).

Also reported: the decode kernel's roofline (algorithmic bytes / event-timed
launch duration against the measured HBM copy bandwidth), the end-to-end
figure through the C ABI with host buffers, the encoder time (also with
GPTQ block compensation), base-3 storage, the prefill (M = 4096) throughput,
the other workloads, and the oracle's CPU time.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
Multi-GPU runs (torchrun, one process per GPU) are independent replicas.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "SDQ-linear decode GB/s vs ~8 TB/s HBM; prefill TOPS vs tensor-core peak"
PROFILE_DECODE = os.path.join(ROOT, "profiles", "decode_llama70b_m1.md")


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5000)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--impl", default="sdq", choices=["sdq", "reference"])
    ap.add_argument("--m", type=int, default=1, help="decode batch")
    ap.add_argument("--no-extras", action="store_true", help="skip encode/prefill/sweep/cpu legs")
    ap.add_argument("--linears", default="", help="comma list of llama-70b-layer linears to run (default: all 7)")
    ap.add_argument("--encode-only", action="store_true",
                    help="run only the base-3 storage and GPTQ encoder legs (for their ncu captures)")
    ap.add_argument("--prefill-only", action="store_true",
                    help="time only the prefill leg (M = 4096) on the chosen linears and print its JSON "
                         "(for profiling the prefill kernels alone)")
    ap.add_argument("--eager", action="store_true",
                    help="launch every step eagerly instead of replaying a CUDA graph (same kernels; "
                         "for profilers that cannot follow stream capture)")
    return ap.parse_args()


# ------------------------------------------------------------------ utils
def max_over_ranks(x, dist):
    """Largest x over all ranks (a job's step time is its slowest rank's)."""
    if not dist:
        return float(x)
    import torch
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([float(x)], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(units_per_rank, world, ms_step):
    """Whole-job throughput (G units / s): what all ranks processed over the step time."""
    return units_per_rank * world / (ms_step * 1e-3) / 1e9


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p["hbm_gbs"], p["bf16_tflops"], p.get("bf16_tflops_sustained", p["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


class ClockSampler:
    """nvidia-smi SM clocks and throttle reasons, sampled every 100 ms."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.idx = gpu_index
        self.rows = []
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
            return
        self.t = threading.Thread(target=self._read, daemon=True)
        self.t.start()

    def _read(self):
        for line in self.proc.stdout:
            self.rows.append((time.time(), line.strip()))

    def stop(self):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self, t0, t1):
        sel = [r for (t, r) in self.rows if t0 - 0.15 <= t <= t1 + 0.15]
        if not sel:
            sel = [r for (_, r) in self.rows[-3:]]
        mhz, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in sel:
            f = [x.strip() for x in r.split(",")]
            try:
                mhz.append(float(f[1]))
                mx = max(mx, float(f[2]))
            except (ValueError, IndexError):
                continue
            for nm, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        mhz.sort()
        med = mhz[len(mhz) // 2] if mhz else None
        return {"sm_mhz": med, "sm_max_mhz": mx or None, "reasons": sorted(reasons),
                "samples": len(sel)}


def code_text(src):
    """C++/CUDA source without comments and empty lines, runs of blanks
    collapsed: the part of a kernel source that a profile depends on."""
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    out = []
    for line in src.splitlines():
        i = line.find("//")
        if i >= 0 and line.count('"', 0, i) % 2 == 0:
            line = line[:i]
        line = " ".join(line.split())
        if line:
            out.append(line)
    return "\n".join(out) + "\n"


def source_hash(src_files):
    h = hashlib.sha256()
    for p in src_files:
        with open(p) as f:
            h.update(code_text(f.read()).encode())
    return h.hexdigest()[:16]


def profile_traffic(src_files):
    """dram bytes per launch from the committed ncu summary, if it was taken
    on the current kernel code (a sha256 of the sources without comments,
    recorded in the summary)."""
    try:
        with open(PROFILE_DECODE) as f:
            txt = f.read()
    except OSError:
        return None, None
    cur = source_hash(src_files)
    vals = {}
    for line in txt.splitlines():
        if ":" in line and line.strip().startswith(("source_sha256", "traffic_bytes_per_launch",
                                                    "traffic_launch_linear")):
            k, v = line.split(":", 1)
            vals[k.strip()] = v.strip()
    if vals.get("source_sha256") != cur:
        return None, cur
    try:
        return int(vals["traffic_bytes_per_launch"]), cur
    except (KeyError, ValueError):
        return None, cur


# ------------------------------------------------------------------ layer
def build_layer(P, W, torch, cfg):
    """Encode + pack every linear of ``cfg`` on the device; returns the plans
    with tiled codes and alpha, and the encode time."""
    layers = []
    enc_ms = 0.0
    for lin in cfg.linears:
        desc = P.LayerDesc(lin.n_out, lin.k_in, cfg.block, lin.osr, cfg.quantizer)
        plan = P.Plan(desc, W.hadamard_signs(lin, cfg.block))
        w = W.weights_device(lin)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        codes, alpha = plan.encode(w)
        tiled = plan.pack(codes)
        e1.record()
        torch.cuda.synchronize()
        enc_ms += e0.elapsed_time(e1)
        del w, codes
        layers.append({"lin": lin, "plan": plan, "tiled": tiled, "alpha": alpha,
                       "code_bytes": P.sdq_tiled_bytes(desc)})
    torch.cuda.empty_cache()
    return layers, enc_ms


def encode_gptq_leg(P, W, torch, cfg):
    """sdq_encode_rows_gptq on every linear of the layer (device weights).
    The factor U of H^-1 (upper triangular, positive diagonal: U^T U = H^-1)
    is drawn directly on the device per input width, outside the timed
    region: the encoder's work does not depend on U's values (the parity
    tests factor a synthetic calibration Hessian instead)."""
    factors = {}
    per = {}
    total = 0.0
    for lin in cfg.linears:
        k = lin.k_in
        if k not in factors:
            g = torch.Generator(device="cuda")
            g.manual_seed(4242 + k)
            u = torch.triu(torch.randn((k, k), generator=g, device="cuda"), diagonal=1) * (0.1 / k ** 0.5)
            u.diagonal().copy_(torch.rand((k,), generator=g, device="cuda") + 0.5)
            factors[k] = u
        desc = P.LayerDesc(lin.n_out, lin.k_in, cfg.block, lin.osr, cfg.quantizer)
        plan = P.Plan(desc, W.hadamard_signs(lin, cfg.block))
        w = W.weights_device(lin)
        codes = plan.alloc_plain()
        alpha = torch.empty(lin.n_out, dtype=torch.float32, device="cuda")
        ws = torch.empty(P.sdq_gptq_workspace_bytes(plan.handle), dtype=torch.uint8, device="cuda")
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        P.sdq_encode_rows_gptq(plan.handle, w, factors[k], codes, alpha, ws)
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1)
        per[lin.name] = round(ms, 2)
        total += ms
        del w, codes, alpha, ws, plan
    del factors
    torch.cuda.empty_cache()
    return {"ms_per_layer": round(total, 1), "per_linear_ms": per,
            "what": "sdq_encode_rows_gptq (encode with GPTQ block compensation), 7 linears; codes bit-exact "
                    "with the oracle's canonical definition"}


def build_group_layers(P, W, torch, cfg):
    """The layer as the linears that share an input (q/k/v, gate/up; see
    workloads.shared_input_groups): one plan per group over the members'
    rows concatenated, with the first member's Hadamard signs; encoded and
    packed on the device.  Each entry's "lin" describes the group's matrix."""
    layers = []
    for name, members in W.shared_input_groups(cfg):
        first = members[0]
        n = sum(m.n_out for m in members)
        desc = P.LayerDesc(n, first.k_in, cfg.block, first.osr, cfg.quantizer)
        plan = P.Plan(desc, W.hadamard_signs(first, cfg.block))
        w = torch.cat([W.weights_device(m) for m in members]) if len(members) > 1 else W.weights_device(first)
        codes, alpha = plan.encode(w)
        tiled = plan.pack(codes)
        torch.cuda.synchronize()
        del w, codes
        lin = W.Linear(name, n, first.k_in, first.osr, first.dist, first.std, first.seed)
        layers.append({"lin": lin, "members": [m.name for m in members], "plan": plan, "tiled": tiled,
                       "alpha": alpha, "code_bytes": P.sdq_tiled_bytes(desc)})
    torch.cuda.empty_cache()
    return layers


def base3_leg(P, torch, layers):
    """Base-3 storage of the layer's codes: bytes against the 2-bit layout and
    the throughput of sdq_pack_base3 / sdq_unpack_base3 (plain <-> base-3;
    bytes read + written per call over the call's time, events)."""
    plain_b = b3_b = 0
    t_pack = t_unpack = 0.0
    for lay in layers:
        plan = lay["plan"]
        d = plan.desc
        plain = plan.alloc_plain()
        P.sdq_unpack(plan.handle, lay["tiled"], plain, None)
        b3 = torch.empty(P.sdq_base3_bytes(d), dtype=torch.uint8, device="cuda")
        back = torch.empty_like(plain)
        for _ in range(2):                                 # warm-up
            P.sdq_pack_base3(plan.handle, plain, b3)
            P.sdq_unpack_base3(plan.handle, b3, back, None)
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        torch.cuda.synchronize()
        ev[0].record()
        P.sdq_pack_base3(plan.handle, plain, b3)
        ev[1].record()
        P.sdq_unpack_base3(plan.handle, b3, back, None)
        ev[2].record()
        torch.cuda.synchronize()
        assert torch.equal(back, plain), "base-3 round trip"
        t_pack += ev[0].elapsed_time(ev[1])
        t_unpack += ev[1].elapsed_time(ev[2])
        plain_b += plain.numel() * 4
        b3_b += b3.numel()
        del plain, b3, back
    torch.cuda.empty_cache()
    gbs = (plain_b + b3_b) / 1e9
    return {"base3_bytes": b3_b, "plain_2bit_bytes": plain_b, "ratio": round(b3_b / plain_b, 4),
            "bits_per_code": 1.6, "pack_GBps": round(gbs / (t_pack * 1e-3), 1),
            "unpack_GBps": round(gbs / (t_unpack * 1e-3), 1),
            "what": "LLaMA-70B layer codes: plain 2-bit <-> base-3 (5 trits per byte), one call per linear; "
                    "GB/s = (plain + base-3 bytes) / time"}


def alg_bytes(lay, M):
    lin = lay["lin"]
    # packed codes (2 bits/code) + alpha + bf16 x + fp32 y
    k_eff = lay["plan"].k_eff
    return lin.n_out * k_eff * 2 // 8 + 4 * lin.n_out + 2 * M * lin.k_in + 4 * M * lin.n_out


def random_plan(P, torch, n, k, block, osr, quantizer, seed):
    """A plan and random valid codes in the tiled layout, drawn on the device
    (timing legs: the contraction's work does not depend on the code values;
    ternary fields 10 are mapped to 00)."""
    from fractions import Fraction
    desc = P.LayerDesc(n, k, block, Fraction(osr), quantizer)
    plan = P.Plan(desc)
    nw = P.sdq_tiled_bytes(desc) // 4
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    w = torch.randint(-2 ** 31, 2 ** 31 - 1, (nw,), generator=g, device="cuda", dtype=torch.int64).to(torch.int32)
    if quantizer == P.SDQ_TERNARY:
        w &= ~(((~w) << 1) & -0x55555556)
    alpha = torch.full((n,), 0.02, dtype=torch.float32, device="cuda")
    return {"plan": plan, "tiled": w, "alpha": alpha, "code_bytes": P.sdq_tiled_bytes(desc), "n": n, "k": k}


def graph_step_ms(torch, stream, calls, reps=50, warm=5):
    """Mean time of one replay of a CUDA graph of `calls` (callables taking
    the stream), events on the replay stream."""
    with torch.cuda.stream(stream):
        for _ in range(2):
            for c in calls:
                c(stream)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for c in calls:
            c(stream)
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        for _ in range(warm):
            g.replay()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(reps):
            g.replay()
        b.record(stream)
    torch.cuda.synchronize()
    return a.elapsed_time(b) / reps


def fwd_call(P, lay, x, y, ws, M):
    return lambda st: P.sdq_linear_forward(lay["plan"].handle, lay["tiled"], lay["alpha"], x, M, y, ws, st)


def step_leg(P, torch, stream, lays, M, reps=50):
    """Decode step over `lays` (one sdq_linear_forward per linear, graph-replayed):
    weight GB/s over the step."""
    calls, keep = [], []
    for lay in lays:
        x = torch.randn(M, lay["k"], device="cuda").to(torch.bfloat16)
        y = torch.empty(M, lay["n"], dtype=torch.float32, device="cuda")
        ws = lay["plan"].alloc_workspace(M)
        keep += [x, y, ws]
        calls.append(fwd_call(P, lay, x, y, ws, M))
    ms = graph_step_ms(torch, stream, calls, reps)
    tot = sum(l["code_bytes"] for l in lays)
    return {"GBps": round(tot / (ms * 1e-3) / 1e9, 1), "us_per_step": round(ms * 1e3, 2),
            "code_bytes_per_step": tot, "calls": len(lays)}


def extra_configs_leg(P, W, torch, stream, hbm):
    """The other workloads, with random device codes: OPT-125M per-linear
    latency (L2 flushed before each call) at M = 1 and 16; the LLaMA-7B layer
    step at M = 1, 4, 16, 64; the LLaMA-13B 4-layer stack under the MultiOSR
    map: M = 8 decode step and M = 2048 prefill (contraction alone and with its
    prepare kernel)."""
    from paper_2510_03275_gb300.multiosr import allocate
    out = {}
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    # OPT-125M
    cfg = W.config(1)
    lat = {}
    for lin in cfg.linears:
        lay = random_plan(P, torch, lin.n_out, lin.k_in, cfg.block, lin.osr, cfg.quantizer, lin.seed)
        for M in (1, 16):
            x = torch.randn(M, lin.k_in, device="cuda").to(torch.bfloat16)
            y = torch.empty(M, lin.n_out, dtype=torch.float32, device="cuda")
            ws = lay["plan"].alloc_workspace(M)
            for _ in range(3):
                P.sdq_linear_forward(lay["plan"].handle, lay["tiled"], lay["alpha"], x, M, y, ws, stream)
            ts = []
            for i in range(15):
                with torch.cuda.stream(stream):
                    flush.fill_(i)
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(stream)
                P.sdq_linear_forward(lay["plan"].handle, lay["tiled"], lay["alpha"], x, M, y, ws, stream)
                b.record(stream)
                torch.cuda.synchronize()
                ts.append(a.elapsed_time(b) * 1e3)
            ts.sort()
            us = ts[len(ts) // 2]
            lat.setdefault(str(M), {})[lin.name] = {"us": round(us, 2),
                                                    "GBps_l2_flushed": round(lay["code_bytes"] / us / 1e3, 1)}
    out["opt125m"] = {"what": "per-linear latency of one sdq_linear_forward (prepare + contraction), L2 "
                              "flushed before each call, median of 15; binary codes, OSR 5/2",
                      "by_batch": lat}
    def grouped(cfg):
        # one plan per group of linears that read the same input (as the headline step)
        return [random_plan(P, torch, sum(m.n_out for m in ms), ms[0].k_in, cfg.block, ms[0].osr, cfg.quantizer,
                            ms[0].seed) for _, ms in W.shared_input_groups(cfg)]

    # LLaMA-7B
    cfg = W.config(2)
    lays = [random_plan(P, torch, l.n_out, l.k_in, cfg.block, l.osr, cfg.quantizer, l.seed) for l in cfg.linears]
    glays = grouped(cfg)
    sweep = {}
    for M in (1, 4, 16, 64):
        r = step_leg(P, torch, stream, glays, M, reps=30)
        r["frac_of_hbm"] = round(r["GBps"] / hbm, 4)
        r["GBps_7_calls"] = step_leg(P, torch, stream, lays, M, reps=30)["GBps"]
        sweep[str(M)] = r
    out["llama7b_layer"] = {"what": "decode step (graph-replayed; 4 plans: q/k/v and gate/up each one plan over "
                                    "their rows, as the headline step; GBps_7_calls: one plan per linear), "
                                    "weight GB/s per batch size",
                            "by_batch": sweep}
    del lays, glays
    # LLaMA-13B 4-layer stack, MultiOSR
    cfg = W.config(3, multiosr=allocate)
    lays = [random_plan(P, torch, l.n_out, l.k_in, cfg.block, l.osr, cfg.quantizer, l.seed) for l in cfg.linears]
    glays = grouped(cfg)
    dec = step_leg(P, torch, stream, glays, 8, reps=10)
    dec["frac_of_hbm"] = round(dec["GBps"] / hbm, 4)
    dec["GBps_28_calls"] = step_leg(P, torch, stream, lays, 8, reps=10)["GBps"]
    del glays
    M = 2048
    ms_k5, ms_all, flops = 0.0, 0.0, 0
    for lay, lin in zip(lays, cfg.linears):
        x = torch.randn(M, lin.k_in, device="cuda").to(torch.bfloat16)
        y = torch.empty(M, lin.n_out, dtype=torch.float32, device="cuda")
        ws = lay["plan"].alloc_workspace(M)
        P.sdq_prep_activations(lay["plan"].handle, x, M, ws, stream)
        P.sdq_contract(lay["plan"].handle, lay["tiled"], lay["alpha"], M, y, ws, stream)
        ms_k5 += graph_step_ms(torch, stream, [lambda st, lay=lay, y=y, ws=ws: P.sdq_contract(
            lay["plan"].handle, lay["tiled"], lay["alpha"], M, y, ws, st)], reps=5, warm=2)
        ms_all += graph_step_ms(torch, stream, [fwd_call(P, lay, x, y, ws, M)], reps=5, warm=2)
        flops += 2 * M * lin.n_out * lay["plan"].k_eff
        del x, y, ws
    out["llama13b_4layers_multiosr"] = {
        "osr": sorted({str(l.osr) for l in cfg.linears}),
        "decode_m8": dec,
        "prefill_m2048": {"tflops_contraction": round(flops / (ms_k5 * 1e-3) / 1e12, 1),
                          "tflops_forward": round(flops / (ms_all * 1e-3) / 1e12, 1),
                          "ms_contraction": round(ms_k5, 3), "ms_forward": round(ms_all, 3),
                          "forward_routes": sorted({P.sdq_forward_route(lay["plan"].handle, M) for lay in lays}),
                          "what": "code-domain flops (2 M N K_eff) per time: the code-domain contraction "
                                  "kernel alone, and sdq_linear_forward as it runs at this batch (route 3: "
                                  "weights rebuilt, then one GEMM; route 2: prepare + contraction)",
                          "flops": flops}}
    del lays, flush
    torch.cuda.empty_cache()
    return out


def measure_decode(P, W, torch, layers, M, args, dist, dev, stream, world, hbm, sample_clocks):
    """The decode step over ``layers`` (one sdq_linear_forward per entry):
    graph-replayed step time, the decode kernel per launch, and the step end
    to end with host buffers."""
    import numpy as np
    code_bytes = sum(l["code_bytes"] for l in layers)
    # per-linear inputs / outputs / workspaces; the step's x and y each live in
    # one buffer (views per linear), so a step moves them with one copy each
    xs = [torch.from_numpy(W.activations(lay["lin"], M).view(np.int16)).view(torch.bfloat16)
          for lay in layers]
    x_all = torch.cat([x.reshape(-1) for x in xs]).cuda()
    y_all = torch.empty(sum(M * lay["lin"].n_out for lay in layers), dtype=torch.float32, device="cuda")
    xo = yo = 0
    for lay in layers:
        lin = lay["lin"]
        lay["x"] = x_all[xo:xo + M * lin.k_in].view(M, lin.k_in)
        lay["y"] = y_all[yo:yo + M * lin.n_out].view(M, lin.n_out)
        xo += M * lin.k_in
        yo += M * lin.n_out
        lay["ws"] = lay["plan"].alloc_workspace(M)
        lay["kernels"] = P.sdq_forward_kernels(lay["plan"].handle, M, lay["x"])

    def step():
        for lay in layers:
            P.sdq_linear_forward(lay["plan"].handle, lay["tiled"], lay["alpha"], lay["x"], M,
                                 lay["y"], lay["ws"], stream)

    # eager warm-up, then capture one step in a CUDA graph
    with torch.cuda.stream(stream):
        for _ in range(3):
            step()
    torch.cuda.synchronize()
    if args.eager:
        replay = step
    else:
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            step()
        torch.cuda.synchronize()
        replay = graph.replay

    sampler = ClockSampler(dev) if sample_clocks else None
    if sampler:
        sampler.start()
        time.sleep(0.3)
    with torch.cuda.stream(stream):
        for _ in range(max(3, args.warmup)):
            replay()
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t_wall0 = time.time()
    ev0.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(args.steps):
            replay()
    ev1.record(stream)
    torch.cuda.synchronize()
    t_wall1 = time.time()
    if dist:
        dist.barrier()
    ms_total = ev0.elapsed_time(ev1)
    clocks = None
    if sampler:
        clocks = sampler.summary(t_wall0, t_wall1)
        sampler.stop()
    ms_total = max_over_ranks(ms_total, dist)
    ms_step = ms_total / args.steps
    value = job_rate(code_bytes, world, ms_step)

    # the decode kernel alone, event-timed per launch, queued back to back
    k_ms, k_bytes = 0.0, 0
    per_lin = []
    reps = 20
    for lay in layers:
        if lay["kernels"] == 2:
            P.sdq_prep_activations(lay["plan"].handle, lay["x"], M, lay["ws"], stream)
    torch.cuda.synchronize()
    # A spin kernel holds the stream while every timed launch is queued, so the
    # events bracket GPU execution only (no host launch gaps).
    with torch.cuda.stream(stream):
        torch.cuda._sleep(int(40e-3 * 2.0e9))
    for rep in range(reps + 3):
        for lay in layers:
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            # the decode kernel as sdq_linear_forward launches it (split-K
            # shares added into y with float reductions), without its
            # prepare kernel: y += result from the prepared workspace
            P.sdq_contract_add(lay["plan"].handle, lay["tiled"], lay["alpha"], M, lay["y"], lay["ws"], stream)
            b.record(stream)
            lay.setdefault("ev", []).append((a, b)) if rep >= 3 else None
    torch.cuda.synchronize()
    for lay in layers:
        d = sum(a.elapsed_time(b) for a, b in lay["ev"]) / len(lay["ev"])
        ab = alg_bytes(lay, M)
        per_lin.append({"linear": lay["lin"].name, "us": round(d * 1e3, 2),
                        "GBps": round(ab / (d * 1e-3) / 1e9, 1)})
        k_ms += d
        k_bytes += ab
    achieved = k_bytes / (k_ms * 1e-3) / 1e9
    srcs = [os.path.join(ROOT, "paper_2510_03275_gb300", "csrc", f) for f in ("decode.cu", "common.cuh")]
    traffic, _ = profile_traffic(srcs)

    # end to end through the C ABI with host buffers (pinned), eager calls
    e2e_steps = min(200, max(20, args.steps // 100))
    hx = x_all.cpu().pin_memory()
    hy = torch.empty_like(y_all, device="cpu").pin_memory()
    h2d = hx.numel() * hx.element_size()
    d2h = hy.numel() * hy.element_size()

    def e2e_step():
        x_all.copy_(hx, non_blocking=True)      # the step's inputs, host -> device
        for lay in layers:
            P.sdq_linear_forward(lay["plan"].handle, lay["tiled"], lay["alpha"], lay["x"], M,
                                 lay["y"], lay["ws"], stream)
        hy.copy_(y_all, non_blocking=True)      # the step's results, device -> host

    with torch.cuda.stream(stream):
        for _ in range(3):
            e2e_step()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        a.record(stream)
        for _ in range(e2e_steps):
            e2e_step()
        b.record(stream)
    torch.cuda.synchronize()
    e2e_ms = a.elapsed_time(b) / e2e_steps
    e2e_val = code_bytes * world / (e2e_ms * 1e-3) / 1e9
    return {"code_bytes": code_bytes, "value": value, "ms_step": ms_step, "clocks": clocks,
            "achieved": achieved, "per_lin": per_lin, "traffic": traffic, "e2e_val": e2e_val,
            "e2e_ms": e2e_ms, "h2d": h2d, "d2h": d2h,
            "kernels": sum(lay["kernels"] for lay in layers)}


def run_sdq(args, rank, world, dist):
    import torch

    import paper_2510_03275_gb300 as P
    from paper_2510_03275_gb300 import workloads as W

    dev = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(dev)
    hbm, tf_burst, tf_sus, peak_src = peaks()
    cfg = W.config(4)
    if args.linears:
        keep = set(args.linears.split(","))
        cfg.linears = [l for l in cfg.linears if l.name in keep]
    M = args.m
    layers, enc_ms = build_layer(P, W, torch, cfg)
    if args.encode_only:
        return {"base3": base3_leg(P, torch, layers), "encode_gptq": encode_gptq_leg(P, W, torch, cfg),
                "config": {"workload": "llama70b-layer encode legs"
                                       + (f" [only {args.linears}]" if args.linears else "")}}
    if args.prefill_only:
        return {"prefill": prefill_leg(P, W, torch, layers, torch.cuda.Stream(), tf_burst, tf_sus, peak_src),
                "config": {"workload": "llama70b-layer prefill, M = 4096"
                                       + (f" [only {args.linears}]" if args.linears else "")}}
    glayers = build_group_layers(P, W, torch, cfg)
    stream = torch.cuda.Stream()
    # headline: the step as 4 calls (q/k/v and gate/up each one plan over
    # their rows: they read the same input); then the 7 linears one call each
    g = measure_decode(P, W, torch, glayers, M, args, dist, dev, stream, world, hbm, sample_clocks=True)
    pl = measure_decode(P, W, torch, layers, M, args, dist, dev, stream, world, hbm, sample_clocks=False)
    code_bytes, value, ms_step, clocks = g["code_bytes"], g["value"], g["ms_step"], g["clocks"]
    achieved, per_lin, traffic = g["achieved"], g["per_lin"], g["traffic"]
    e2e_val, e2e_ms, h2d, d2h = g["e2e_val"], g["e2e_ms"], g["h2d"], g["d2h"]

    out = {
        "metric": METRIC, "value": round(value, 1), "unit": "GB/s",
        "n_gpus": world, "steps": args.steps, "warmup": max(3, args.warmup),
        "ms_per_step": round(ms_step, 5), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "u2-codes/e2m1-mma(mxf4)/f32-acc", "data": "synthetic",
        "config": {"workload": "llama70b-layer decode: q/o 8192x8192, k/v 1024x8192, "
                               "gate/up 28672x8192, down 8192x28672; OSR 2 ternary B=128"
                               + (f" [only {args.linears}]" if args.linears else ""),
                   "calls_per_step": len(glayers),
                   "plans": [f"{lay['lin'].name} {lay['lin'].n_out}x{lay['lin'].k_in} = "
                             + "+".join(lay["members"]) for lay in glayers],
                   "grouping": "linears that read the same input (q/k/v, gate/up) as one plan over their "
                               "rows: per-row codes and alpha make each member's outputs those of its own plan",
                   "decode_batch": M, "code_bytes_per_step": code_bytes,
                   "l2": "7 code matrices (428 MB) streamed in turn > 129 MB L2",
                   "timing": ("eager launches" if args.eager else "CUDA graph of one step, replayed")
                             + "; events on the launch stream",
                   "parallelism": f"replicas x{world}"},
        "clocks": clocks,
        "e2e": {"value": round(e2e_val, 1), "unit": "GB/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "ms_per_step": round(e2e_ms, 4),
                "how": "per step: one pinned-host -> device copy of all x, eager sdq_linear_forward "
                       "per linear, one device -> pinned-host copy of all y"},
        "gpu_launches": g["kernels"] * args.steps,
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": hbm,
                     "unit": "GB/s", "frac": round(achieved / hbm, 4), "traffic": traffic,
                     "kernel": f"decode_kernel, per launch as in the step (sdq_contract_add on the prepared "
                               f"workspace, M={M}; the 4 plans of the step)",
                     "peak_source": peak_src,
                     "nominal_8tbs_frac": round(achieved / 8000.0, 4), "per_linear": per_lin},
        "roofline_per_step": {"bound": "hbm", "achieved": round(value, 1), "peak": hbm, "unit": "GB/s",
                              "frac": round(value / hbm, 4),
                              "what": "code bytes of the step / step time: both kernels of every call "
                                      "and the gaps between them"},
        "encode": {"ms_per_layer": round(enc_ms, 3), "what": "sdq_encode_rows + sdq_pack, 7 linears"},
    }
    out["per_linear_step"] = {
        "GBps": round(pl["value"], 1), "frac_of_hbm": round(pl["value"] / hbm, 4),
        "ms_per_step": round(pl["ms_step"], 5), "calls": len(layers),
        "per_launch": {"achieved": round(pl["achieved"], 1), "frac": round(pl["achieved"] / hbm, 4),
                       "per_linear": pl["per_lin"]},
        "e2e_GBps": round(pl["e2e_val"], 1),
        "what": "the same layer as 7 calls, one plan per linear (each with its own Hadamard signs)"}
    if not args.no_extras and rank == 0:
        out["decode_sweep"] = decode_sweep(P, W, torch, glayers, stream, hbm, tf_burst, peak_src)
        out["decode_sweep"]["values_7_calls"] = decode_sweep(P, W, torch, layers, stream, hbm, tf_burst,
                                                             peak_src)["values"]
        out["other_configs"] = extra_configs_leg(P, W, torch, stream, hbm)
        out["prefill"] = prefill_leg(P, W, torch, layers, stream, tf_burst, tf_sus, peak_src)
        out["base3"] = base3_leg(P, torch, layers)
        out["encode_gptq"] = encode_gptq_leg(P, W, torch, W.config(4))
        out["cpu_baseline"] = cpu_baseline_leg()
        try:
            out["encode"]["cpu"] = encode_cpu_leg()
        except Exception as e:   # a reported comparison only: never fail the run on it
            out["encode"]["cpu"] = {"unavailable": f"{type(e).__name__}: {e}"[:200]}
    return out


def sweep_roofline(code_bytes, ops, ms, hbm_gbs, fp8_tflops):
    """Bound and fraction of one batch size of the decode sweep: the time the
    codes need at the HBM peak against the time the algorithmic add/sub work
    (2 M N K_eff flop-equivalents) needs at the fp8 tensor peak; whichever is
    longer is the bound, and frac = that time / the measured time."""
    t_hbm = code_bytes / (hbm_gbs * 1e9)
    t_ten = ops / (fp8_tflops * 1e12)
    bound, t = ("hbm", t_hbm) if t_hbm >= t_ten else ("tensor", t_ten)
    return {"bound": bound, "frac": round(t / (ms * 1e-3), 4)}


def decode_sweep(P, W, torch, layers, stream, hbm_gbs, tf_bf16, peak_src):
    import numpy as np
    res, roof = {}, {}
    fp8 = 2.0 * tf_bf16   # e4m3 dense peak: the measured bf16 peak x the nominal 2x ratio
    for M in (1, 2, 4, 8, 16, 32, 64):
        tot_b, tot_ms, tot_ops = 0, 0.0, 0.0
        for lay in layers:
            lin = lay["lin"]
            x = torch.from_numpy(W.activations(lin, M).view(np.int16)).view(torch.bfloat16).cuda()
            y = torch.empty((M, lin.n_out), dtype=torch.float32, device="cuda")
            ws = lay["plan"].alloc_workspace(M)
            for _ in range(3):
                P.sdq_linear_forward(lay["plan"].handle, lay["tiled"], lay["alpha"], x, M, y, ws, stream)
            evs = []
            torch.cuda.synchronize()
            with torch.cuda.stream(stream):
                torch.cuda._sleep(int(5e-3 * 2.0e9))   # queue the timed launches behind a spin
            for _ in range(10):
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(stream)
                P.sdq_linear_forward(lay["plan"].handle, lay["tiled"], lay["alpha"], x, M, y, ws, stream)
                b.record(stream)
                evs.append((a, b))
            torch.cuda.synchronize()
            tot_ms += sum(a.elapsed_time(b) for a, b in evs) / len(evs)
            tot_b += lay["code_bytes"]
            tot_ops += 2.0 * M * lin.n_out * lay["plan"].k_eff
        res[str(M)] = round(tot_b / (tot_ms * 1e-3) / 1e9, 1)
        roof[str(M)] = sweep_roofline(tot_b, tot_ops, tot_ms, hbm_gbs, fp8)
    return {"unit": "weight GB/s (sdq_linear_forward per plan of the step, inputs on the device, per batch "
                    "size; values_7_calls: one plan per linear)",
            "values": res, "roofline": roof,
            "peaks": {"hbm_gbs": hbm_gbs, "fp8_tflops": fp8,
                      "source": peak_src + " (fp8 = bf16 x 2, nominal ratio)"}}


def prefill_leg(P, W, torch, layers, stream, tf_burst, tf_sus, peak_src):
    """M = 4096 over the 7 linears: the code-domain contraction kernel alone
    (its roofline), the code-domain route with its prepare kernel, and
    sdq_linear_forward as it runs at this batch (the dense route where the
    plan allows it: weights rebuilt, then one GEMM)."""
    import numpy as np
    M = 4096
    flops, exe, ms, ms_p, ms_f = 0, 0, 0.0, 0.0, 0.0
    routes = set()

    def timed(fn, n=5):
        evs = []
        for _ in range(n):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            fn()
            b.record(stream)
            evs.append((a, b))
        return evs

    try:
        for lay in layers:
            lin = lay["lin"]
            h = lay["plan"].handle
            x = torch.from_numpy(W.activations(lin, M).view(np.int16)).view(torch.bfloat16).cuda()
            y = torch.empty((M, lin.n_out), dtype=torch.float32, device="cuda")
            ws = lay["plan"].alloc_workspace(M)
            P.sdq_prep_activations(h, x, M, ws, stream)
            P.sdq_contract(h, lay["tiled"], lay["alpha"], M, y, ws, stream)
            P.sdq_linear_forward(h, lay["tiled"], lay["alpha"], x, M, y, ws, stream)
            evs = timed(lambda: P.sdq_contract(h, lay["tiled"], lay["alpha"], M, y, ws, stream))
            evp = timed(lambda: (P.sdq_prep_activations(h, x, M, ws, stream),
                                 P.sdq_contract(h, lay["tiled"], lay["alpha"], M, y, ws, stream)))
            evf = timed(lambda: P.sdq_linear_forward(h, lay["tiled"], lay["alpha"], x, M, y, ws, stream))
            torch.cuda.synchronize()
            ms += sum(a.elapsed_time(b) for a, b in evs) / len(evs)
            ms_p += sum(a.elapsed_time(b) for a, b in evp) / len(evp)
            ms_f += sum(a.elapsed_time(b) for a, b in evf) / len(evf)
            keff = lay["plan"].k_eff
            flops += 2 * M * lin.n_out * keff
            route = P.sdq_forward_route(h, M)
            routes.add(route)
            # executed tensor work of the route sdq_linear_forward takes: the
            # dense GEMM plus the rebuild (hi and lo parts of G), or the
            # code-domain contraction plus the prepare GEMM (hi and lo)
            b_ = W.config(4).block
            exe += (2 * M * lin.n_out * lin.k_in + 4 * lin.n_out * keff * b_) if route == 3 \
                else (2 * M * lin.n_out * keff + 4 * M * keff * b_)
            del x, y, ws
    except P.SdqError as e:
        return {"unavailable": str(e)}
    tflops = flops / (ms * 1e-3) / 1e12
    names = {1: "decode", 2: "code domain (prepare + contraction)", 3: "dense (weights rebuilt, then one GEMM)"}
    return {"value": round(tflops, 1), "unit": "TFLOP/s", "M": M, "ms_per_layer": round(ms, 3),
            "flops_per_layer": flops,
            "what": "the code-domain contraction kernel alone (sdq_contract), 2 M N K_eff flops",
            "with_prepare": {"value": round(flops / (ms_p * 1e-3) / 1e12, 1), "unit": "TFLOP/s",
                             "ms_per_layer": round(ms_p, 3),
                             "what": "code-domain route: sdq_prep_activations (x_tilde in bf16) + sdq_contract"},
            "forward": {"route": " / ".join(names[r] for r in sorted(routes)),
                        "ms_per_layer": round(ms_f, 3),
                        "code_domain_tflops": round(flops / (ms_f * 1e-3) / 1e12, 1),
                        "executed_flops_per_layer": exe,
                        "executed_tflops": round(exe / (ms_f * 1e-3) / 1e12, 1),
                        "frac_of_bf16_peak": round(exe / (ms_f * 1e-3) / 1e12 / tf_burst, 4),
                        "what": "sdq_linear_forward as it runs at M = 4096; code_domain_tflops = the "
                                "code-domain flops (2 M N K_eff) / its time, executed_tflops = the tensor "
                                "work its route performs / its time"},
            "roofline": {"bound": "tensor", "achieved": round(tflops, 1), "peak": tf_burst,
                         "unit": "TFLOP/s", "frac": round(tflops / tf_burst, 4),
                         "peak_source": peak_src + " bf16 burst"}}


# -------------------------------------------------------- oracle (CPU) legs
class OracleSample:
    """Seeded inputs for the oracle's code-domain forward (decode, M=1) on
    `rows` rows of every llama-70b-layer linear, prepared once; `run()` times one pass."""

    def __init__(self, rows):
        import numpy as np

        from paper_2510_03275_gb300 import workloads as W
        cfg = W.config(4)
        self.items = []
        self.nbytes = 0
        for lin in cfg.linears:
            nb = cfg.n_b(lin)
            keff = lin.k_in // cfg.block * nb
            codes = W.random_codes(rows, keff, cfg.quantizer, seed=lin.seed)
            alpha = np.full(rows, 0.02, dtype=np.float32)
            x = W.bf16_to_float(W.activations(lin, 1))
            self.items.append((x, codes, alpha, cfg.block, nb, W.hadamard_signs(lin, cfg.block)))
            self.nbytes += rows * keff * 2 // 8

    def run(self):
        import oracle as O
        t0 = time.perf_counter()
        for x, codes, alpha, block, nb, signs in self.items:
            O.forward_code_domain(x, codes, alpha, block, nb, signs)
        return time.perf_counter() - t0


def _cores():
    return len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()


def _host_threads():
    """The host the oracle runs on: logical CPUs, the ones this process may
    use, and the BLAS thread pools numpy would use (threadpoolctl when it is
    installed, else the environment's thread settings)."""
    import numpy  # noqa: F401  (loads the BLAS whose pools are reported)
    info = {"cpu_count": os.cpu_count(), "affinity": _cores()}
    pools = []
    try:
        from threadpoolctl import threadpool_info
        pools = [{"api": d.get("internal_api"), "threads": d.get("num_threads")} for d in threadpool_info()]
    except Exception:
        pass
    info["blas"] = pools or {k: os.environ.get(k, "unset") for k in
                             ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")}
    return info


def cpu_baseline_leg(sample_rows=256, min_secs=10.0):
    """The oracle timed on the host cores: repeated passes over a bounded
    sample until about `min_secs` of CPU work."""
    smp = OracleSample(sample_rows)
    secs, passes = 0.0, 0
    while secs < min_secs:
        secs += smp.run()
        passes += 1
    cores = _cores()
    return {"value": round(smp.nbytes * passes / secs / 1e9, 4), "unit": "GB/s", "cores": cores,
            "kind": "oracle", "host": _host_threads(),
            "sample": f"oracle forward_code_domain (fp64 numpy), decode M=1, {sample_rows} rows of "
                      f"each of the 7 llama-70b-layer linears ({smp.nbytes} code bytes) x {passes} passes = "
                      f"{secs:.1f} s; numpy default threads on {cores} host cores"}


def encode_cpu_leg(rows=64):
    """The oracle's canonical fp32 encoder (the bit-exact contract of
    sdq_encode_rows) timed on the host on the first `rows` rows of every
    llama-70b-layer linear, extrapolated linearly to the full layer and
    labelled as such."""
    import numpy as np
    import oracle as O
    from paper_2510_03275_gb300 import workloads as W
    cfg = W.config(4)
    secs = 0.0
    for lin in cfg.linears:
        w = W.weights(lin, rows=np.arange(rows))
        signs = W.hadamard_signs(lin, cfg.block)
        nb = int(cfg.block * lin.osr)
        t0 = time.perf_counter()
        O.encode(w, cfg.block, nb, cfg.quantizer, O.ALPHA_MAXABS, signs)
        secs += (time.perf_counter() - t0) * lin.n_out / rows
    return {"oracle_ms_per_layer_extrapolated": round(secs * 1e3, 1), "cores": _cores(),
            "sample": f"oracle encode (canonical fp32, numpy) on {rows} rows of each of the 7 "
                      "linears, scaled by rows to the full layer"}


def run_reference(args, rank, world):
    """The oracle as the reference arm: each step is the code-domain forward on
    a bounded row sample of every llama-70b-layer linear (GB/s of codes processed)."""
    if rank != 0:
        return None
    rows = 64 if args.steps <= 2000 else 16
    smp = OracleSample(rows)
    warm = max(3, args.warmup)
    for _ in range(warm):
        smp.run()
    secs = 0.0
    for _ in range(args.steps):
        secs += smp.run()
    val = smp.nbytes * args.steps / secs / 1e9
    cores = _cores()
    return {"impl": "reference", "metric": METRIC, "value": round(val, 4), "unit": "GB/s",
            "n_gpus": world, "steps": args.steps, "warmup": warm,
            "ms_per_step": round(secs / args.steps * 1e3, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": "llama70b-layer decode, M=1; oracle on a bounded "
                                   f"sample of {rows} rows per linear per step"},
            "cpu_baseline": {"value": round(val, 4), "unit": "GB/s", "cores": cores,
                             "kind": "oracle", "host": _host_threads(),
                             "sample": f"{rows} rows of each of the 7 llama-70b-layer linears per step"},
            "e2e": {"value": round(val, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def main():
    args = parse()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    dist = None
    if world > 1:
        import torch
        import torch.distributed as td
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if torch.cuda.is_available():
            torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
        td.init_process_group(backend)
        dist = td
    if args.impl == "reference":
        out = run_reference(args, rank, world)
    else:
        out = run_sdq(args, rank, world, dist)
    if rank == 0 and out is not None:
        print(json.dumps(out))
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
