"""The N > 1 paths on the CPU (gloo, world size 2): the replicas-only aggregation of bench.py (no
data-path collective: each rank runs its own replica; the job's step time is the slowest rank's,
and the job's throughput counts every rank's work) and the reference arm launched the way the
driver launches a multi-GPU bench (rank 0 alone runs and prints; the other ranks exit 0)."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _replica(rank, world, port, out):
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    step_ms = 1.0 + rank                           # rank 1 is the slower replica
    slowest = bench.reduce_max(step_ms, world, "cpu")
    value = bench.job_throughput(1e12, world, slowest)
    dist.barrier()
    out.put((rank, slowest, value))
    dist.destroy_process_group()


def test_replica_aggregation_on_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_replica, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(out.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    # both ranks see the slowest step (2 ms); the job does 2 x 1e12 ops per 2 ms = 1000 TOPS
    assert [r[1] for r in res] == [2.0, 2.0]
    assert all(abs(r[2] - 1000.0) < 1e-9 for r in res)


def test_reference_arm_under_torchrun_two_ranks():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py", "--impl", "reference",
           "--gpus", "2", "--steps", "2", "--warmup", "3"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600,
                       env=dict(os.environ, OMP_NUM_THREADS="1"))
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"


def test_profiled_traffic_is_keyed_by_workload_and_kernel_source(tmp_path, monkeypatch):
    """bench.py reports an ncu DRAM-traffic figure only from a summary taken on the same workload
    and on the kernel source as it stands (a stale or foreign figure is null)."""
    sys.path.insert(0, ROOT)
    import bench
    sha = bench.kernel_sha()
    (tmp_path / "conv_tc_a.md").write_text(f"# a\n\nworkload: wl_a\nkernel_sha: {sha}\ntraffic_bytes_per_launch: 123\n")
    (tmp_path / "conv_tc_b.md").write_text("# b\n\nworkload: wl_b\nkernel_sha: 0000000000000000\n"
                                           "traffic_bytes_per_launch: 456\n")
    monkeypatch.setattr(bench, "PROFILES", str(tmp_path))
    assert bench.profiled_traffic("wl_a") == 123.0
    assert bench.profiled_traffic("wl_b") is None        # taken on another kernel source
    assert bench.profiled_traffic("wl_c") is None        # no summary for this workload


def test_bench_counts_the_resnet18_step_ops_and_algorithmic_bytes():
    """bench.py's ops (2 per MAC) and algorithmic bytes of the ResNet-18 body at batch 32, against
    the network written out layer by layer here: 108.5 GOP and 31.2 MB per step."""
    sys.path.insert(0, ROOT)
    import bench
    from paper_1911_08076_gb300 import synth
    B = 32
    # (input size, cin, cout, k, stride) of the 19 convs
    layers = [(56, 64, 64, 3, 1)] * 4
    for c_in, c, h in ((64, 128, 56), (128, 256, 28), (256, 512, 14)):
        layers += [(h, c_in, c, 3, 2), (h, c_in, c, 1, 2)] + [(h // 2, c, c, 3, 1)] * 3
    ops = nbytes = 0
    for h, cin, cout, k, s in layers:
        ho = h // s
        ops += 2 * B * ho * ho * cout * k * k * cin
        nbytes += B * h * h * cin / 4 + k * k * cin * cout / 8 + 13 * cout + B * ho * ho * cout / 4
    wl = synth.get("resnet18")
    convs = [l for l in wl.layers if l.kind == "conv"]
    assert len(convs) == 19
    assert abs(sum(bench.conv_ops(l, B) for l in convs) - ops) < 1
    assert abs(sum(bench.alg_bytes(l, B, 2) for l in convs) - nbytes) < 1
    assert round(ops / 1e9, 1) == 108.5 and round(nbytes / 1e6, 1) == 31.2
