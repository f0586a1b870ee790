"""N > 1 path of bench.py on the CPU with the gloo backend (world size 2):
the step time is the slowest rank's, the job's value counts every rank's
units, and under torchrun only rank 0 prints the reference arm's line.
Replicas only: the decode path has no exchange step, so there is no
collective on the data path to test."""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, values, out):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    out[rank] = bench.max_over_ranks(values[rank], dist)
    dist.barrier()
    dist.destroy_process_group()


def test_max_over_ranks_gloo_world2():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    vals = [3.25, 7.5]
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, vals, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    assert dict(out) == {0: 7.5, 1: 7.5}


def test_job_rate_counts_all_ranks():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.job_rate(1e9, 1, 1000.0) == pytest.approx(1.0)
    assert bench.job_rate(1e9, 4, 1000.0) == pytest.approx(4.0)
    assert bench.max_over_ranks(2.5, None) == 2.5


def test_sweep_roofline_bound_and_fraction():
    """Per-batch decode roofline: the longer of the HBM time of the codes and
    the fp8 tensor time of the 2 M N K_eff add/sub work bounds the batch."""
    sys.path.insert(0, ROOT)
    import bench
    # 1 GB of codes at 1000 GB/s = 1 ms; 2 GFLOP at 1 TFLOP/s = 2 ms; measured 4 ms
    assert bench.sweep_roofline(1e9, 2e9, 4.0, 1000.0, 1.0) == {"bound": "tensor", "frac": 0.5}
    assert bench.sweep_roofline(1e9, 0.5e9, 2.0, 1000.0, 1.0) == {"bound": "hbm", "frac": 0.5}
    # the LLaMA-70B layer at M = 64 against this pool's peaks is still HBM-bound
    codes, ops = 427819008, 2.0 * 64 * 427819008 * 4   # 4 codes per byte (2-bit ternary)
    r = bench.sweep_roofline(codes, ops, 1.0, 6783.5, 2 * 1903.9)
    assert r["bound"] == "hbm"


def test_profile_hash_ignores_comments_only():
    """The ncu summary stays valid across comment edits of the kernel source,
    not across code edits (a string holding // is code)."""
    sys.path.insert(0, ROOT)
    import bench
    a = 'int f() {  // note\n  /* block\n comment */ return 1;\n}\n'
    b = '// header\nint f() {\n\n  return 1;   \n}\n'
    assert bench.code_text(a) == bench.code_text(b)
    assert bench.code_text('int g = 2;\n') != bench.code_text('int g = 3;\n')
    assert "//x" in bench.code_text('const char* s = "//x";\n')


def test_encode_cpu_leg_extrapolates():
    """The host-side encode timing of the bench: a positive per-layer figure
    from a row sample (CPU only)."""
    sys.path.insert(0, ROOT)
    import bench
    r = bench.encode_cpu_leg(rows=2)
    assert r["oracle_ms_per_layer_extrapolated"] > 0 and r["cores"] >= 1 and "2 rows" in r["sample"]


def test_reference_arm_under_torchrun_world2():
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr=127.0.0.1", f"--master-port={_free_port()}", "bench.py",
           "--impl", "reference", "--gpus", "2", "--steps", "2", "--warmup", "3"]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1                      # rank 0 alone prints
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle"
