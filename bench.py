#!/usr/bin/env python
"""Throughput benchmark of the quantized-substructure path on GB300.

A step is one pass of a layer stack over one batch through ifq_forward, replayed
as a CUDA graph.  The headline workload is the largest single-GPU configuration:
the 3x3 256->256 binary x 2-bit conv at 56x56, batch 256 (GEMM M = 802816,
N = 256, K = 2304, 947 GOP).  The same JSON line carries a sub-record for every
other configuration (the single PR1 layer, the ResNet-18 body b32, AlexNet
conv2-FC7 b128, Tiny-YOLO and Tinier-YOLO b64 with fused pools, IFQ-Tinier-YOLO
end to end from 8-bit pixels, the 1x1 512->512 layer b256), each with its step
time, TOPS, images/s, roofline fraction, per-layer times, end-to-end figure and
the oracle's CPU baseline.

Inputs are seeded synthetic codes already resident in HBM; L2 is flushed (a
256 MB write) between timed steps, outside the per-step CUDA events.  `e2e`
replays a graph from ifq_graph_create_io that also copies the pinned host input
in and every result out, one launch per step.  `roofline` is the conv kernel
against the measured tensor peak (MEASURED_PEAKS.json bf16 x 2), with the DRAM
traffic of the committed ncu summary of the same workload and kernel source;
beside it, fractions against the e4m3 tcgen05 and the s8 mma.sync rates
measured in the same process.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference] [--workload NAME] [--no-sub]

Rank 0 prints one JSON line.  Under torchrun each rank runs an independent
replica (no data-path collective; a barrier and a max over ranks time the job).
`--impl reference` times the CPU oracle on the host cores on bounded samples
of the same workload.
"""
from __future__ import annotations

import argparse
import ctypes
import glob
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_1911_08076_gb300 import synth  # noqa: E402

METRIC = "binary×2-bit conv TOPS and images/s at 1 GB300; % of dense INT8 peak"
UNIT = "TOPS"
HEADLINE = "roofline3x3"
SUB_WORKLOADS = ["pr1", "resnet18", "alexnet", "tinyyolo_fused", "tinieryolo_fused", "tinieryolo_full_fused",
                 "roofline1x1"]
FP8_PER_BF16 = 2.0          # nominal dense fp8 / bf16 tensor ratio (4.5 / 2.25 PFLOP/s)
FALLBACK_BF16_TFLOPS = 1900.0
PROFILES = os.path.join(ROOT, "profiles")
KERNEL_DIR = os.path.join(ROOT, "paper_1911_08076_gb300", "csrc")
RATES_SRC = os.path.join(ROOT, "bench_rates.cu")
RATES_LIB = os.path.join(ROOT, "_build", "libbench_rates.so")


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def dist_info():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)),
            int(os.environ.get("LOCAL_RANK", 0)))


def conv_ops(layer, batch):
    return 2.0 * batch * layer.ho * layer.wo * layer.cout * layer.k * layer.k * layer.cin


def alg_bytes(layer, batch, kbits=2):
    """Bytes the method must move for one conv launch: input codes read once (f/8 bytes per code,
    f = 2 for k = 2 and 4 for k = 3, 4), 1-bit filters, 4 (2^k - 1) + 1 bytes of thresholds and
    sign per channel, output codes at f bits (int32 for accumulators), after the fused pool when
    the launch has one."""
    cb = synth.field_bits(kbits) / 8
    inp = batch * layer.h * layer.w * layer.cin * (1 if getattr(layer, "in_bits", 0) == 8 else cb)
    wts = layer.cout * layer.k * layer.k * layer.cin / 8
    thr = (4 * ((1 << kbits) - 1) + 1) * layer.cout
    out = batch * layer.out_h * layer.out_w * layer.cout
    out = out * cb if layer.out == "codes" else (out * 4 if layer.out == "acc" else out * (4 + cb))
    return inp + wts + thr + out


def layer_alg_bytes(wl, li, batch):
    """Algorithmic bytes of any layer of a stack: a conv as alg_bytes; a code pool reads its input
    and writes its output once; a fixed-point output reads and writes one int32 per value."""
    l = wl.layers[li]
    if l.kind == "conv":
        return alg_bytes(l, batch, wl.kbits)
    cb = synth.field_bits(wl.kbits) / 8
    if l.kind == "pool":
        return batch * l.c * (l.h * l.w + l.ho * l.wo) * cb
    s = wl.layers[l.src]
    return 2 * 4 * batch * s.out_h * s.out_w * s.cout


def read_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return float(p["bf16_tflops"]), float(p.get("bf16_tflops_sustained", p["bf16_tflops"])), \
            float(p["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_BF16_TFLOPS, 1700.0, 6800.0, "fallback"


def kernel_sha():
    """Hash of every CUDA source of the library (all .cu and .cuh files), so that a change to any
    kernel a workload launches marks its ncu summary stale and its traffic is not reused."""
    h = hashlib.sha256()
    for path in sorted(glob.glob(os.path.join(KERNEL_DIR, "*.cu")) + glob.glob(os.path.join(KERNEL_DIR, "*.cuh"))):
        h.update(os.path.basename(path).encode())
        with open(path, "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(workload: str):
    """DRAM bytes per conv launch from the committed ncu summary of this workload, if it was taken
    on this kernel source (a summary names its `workload:` and `kernel_sha:`)."""
    for path in sorted(glob.glob(os.path.join(PROFILES, "*.md"))):
        try:
            txt = open(path).read()
        except OSError:
            continue
        wl = re.search(r"^workload:\s*(\S+)", txt, re.M)
        sha = re.search(r"^kernel_sha:\s*([0-9a-f]+)", txt, re.M)
        tb = re.search(r"^traffic_bytes_per_launch:\s*([0-9.eE+]+)", txt, re.M)
        if wl and sha and tb and wl.group(1) == workload and sha.group(1) == kernel_sha():
            return float(tb.group(1))
    return None


def build_rates(force: bool = False) -> str:
    """Compile bench_rates.cu (the instruction-rate probes) into _build/libbench_rates.so."""
    if not force and os.path.exists(RATES_LIB) and os.path.getmtime(RATES_LIB) >= os.path.getmtime(RATES_SRC):
        return RATES_LIB
    from paper_1911_08076_gb300 import build as B
    os.makedirs(os.path.dirname(RATES_LIB), exist_ok=True)
    tmp = RATES_LIB + f".{os.getpid()}.tmp"
    nvcc = B._nvcc()
    cudalib = os.path.join(os.path.dirname(os.path.dirname(nvcc)), "lib64")
    subprocess.check_call([nvcc, *B.ARCH, "-O3", "-std=c++17", "-Xcompiler", "-fPIC", "-shared", "-cudart", "shared",
                           RATES_SRC, "-Xlinker", f"-rpath={cudalib}", "-o", tmp])
    os.replace(tmp, RATES_LIB)
    return RATES_LIB


def measure_rates(stream):
    """Tensor rates measured now, on this GPU: tcgen05 e4m3 at N = 128 and 256 (the conv's
    instruction) and mma.sync s8 (the dense INT8 path)."""
    try:
        L = ctypes.CDLL(build_rates())
    except Exception as e:  # no nvcc or no library: report the reason, not a guess
        return {"error": f"rate probes unavailable: {e}"}
    dbl = ctypes.c_double
    L.bench_tc_e4m3_tops.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_void_p, ctypes.POINTER(dbl)]
    L.bench_mma_s8_tops.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_void_p, ctypes.POINTER(dbl)]
    out = {}
    L.bench_tc_e4m3_tops_a.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_void_p,
                                       ctypes.POINTER(dbl)]
    for n in (128, 256):
        v = dbl(0.0)
        rc = L.bench_tc_e4m3_tops(n, 8192, 5, ctypes.c_void_p(stream.cuda_stream), ctypes.byref(v))
        out[f"tcgen05_e4m3_n{n}_tops"] = v.value if rc == 0 else None
    v = dbl(0.0)
    rc = L.bench_tc_e4m3_tops_a(128, 1, 8192, 5, ctypes.c_void_p(stream.cuda_stream), ctypes.byref(v))
    out["tcgen05_e4m3_tmem_a_n128_tops"] = v.value if rc == 0 else None
    v = dbl(0.0)
    rc = L.bench_mma_s8_tops(4096, 3, ctypes.c_void_p(stream.cuda_stream), ctypes.byref(v))
    out["mma_sync_s8_tops"] = v.value if rc == 0 else None
    out["how"] = ("same process, before the timed regions: one CTA per SM issuing M128xNxK32 e4m3 tcgen05 MMAs "
                  "back to back (A in shared memory; tmem_a: A in tensor memory, as the conv issues them); "
                  "4 CTAs x 8 warps per SM issuing m16n8k32 s8 mma.sync; 2 ops per MAC")
    return out


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu_id = gpu_id
        self.proc = None
        self.out = None

    def start(self):
        try:
            self.out = tempfile.TemporaryFile(mode="w+")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", self.gpu_id, f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=self.out, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception as e:  # no nvidia-smi: report nothing rather than guess
            log("clock sampler unavailable:", e)
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.1)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.out.seek(0)
        rows = [l.strip().split(", ") for l in self.out.read().splitlines() if l.strip()]
        sm, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in rows:
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                mx.append(float(r[2]))
            except ValueError:
                continue
            for n, v in zip(names, r[5:9]):
                if v.strip().lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def line_config(wl, args):
    """The `config` object of both arms' JSON lines (identical for the same workload)."""
    convs = [l for l in wl.layers if l.kind == "conv"]
    return {"workload": wl.name, "batch_per_gpu": wl.batch, "layers": len(wl.layers),
            "ops_per_step": sum(conv_ops(l, wl.batch) for l in convs),
            "parallelism": f"replicas x{args.gpus}" if args.gpus > 1 else "single GPU",
            "l2": "flushed between steps (256 MB write outside the step events)", "path": args.path}


def cpu_baseline(wl, x, params, seconds: float):
    """The oracle as it stands (float and integer chains, naive loops) on the host cores, on whole
    images of the workload, images split across threads: as many images as fit in about
    `seconds` of host time (at least one), scaled to the workload's metric."""
    from oracle import oracle as O
    O.build()
    threads = len(os.sched_getaffinity(0))
    per_img = sum(conv_ops(l, 1) for l in wl.layers if l.kind == "conv")
    n_done, dt, n = 0, 0.0, threads   # one image per host thread to start with
    while dt < seconds and n_done < wl.batch:
        n = min(n, wl.batch - n_done)
        t0 = time.perf_counter()
        O.forward(wl, x[n_done:n_done + n], params, threads=threads)
        dt += time.perf_counter() - t0
        n_done += n
        rate = n_done / dt if dt > 0 else 1.0
        n = max(1, min(4 * n, int(rate * max(seconds - dt, 0.0))))
    ops = n_done * per_img
    return {"value": ops / dt / 1e12, "unit": UNIT, "cores": threads, "kind": "oracle",
            "sample": f"{n_done} of the {wl.batch} images of the batch through all {len(wl.layers)} layers, "
                      f"float and integer chains, {dt:.2f} s wall", "images_per_s": n_done / dt}


def run_reference(args):
    """CPU oracle arm: each step is one bounded sample of the workload (a slice of the output
    channels of one conv layer for one image, cycling through the layers), sized so that the
    whole run stays within a few minutes for any --steps/--warmup."""
    rank, world, _ = dist_info()
    if rank != 0:
        return
    from concurrent.futures import ThreadPoolExecutor
    from oracle import oracle as O
    O.build()
    wl = synth.get(args.workload, args.batch)
    x, params = synth.draw_workload(wl, batch=1)
    outs = O.forward(wl, x, params, images=[0], check_float=False)
    convs = [i for i, l in enumerate(wl.layers) if l.kind == "conv"]
    threads = len(os.sched_getaffinity(0))
    inputs, folded = {}, {}
    for li in convs:
        l = wl.layers[li]
        src = x[0:1] if l.src < 0 else outs[l.src]
        inputs[li] = src["codes"] if isinstance(src, dict) else src
        p = O.Params.from_synth(params[li], wl.kbits)
        folded[li] = (p,) + O.fold(p, O.fold_k(l) if wl.kbits == 2 else l.k * l.k * l.cin)
    # calibrate the oracle's rate (MAC/s per thread) on a few channels of the first layer
    l0 = wl.layers[convs[0]]
    t0 = time.perf_counter()
    O.conv_acc(inputs[convs[0]], params[convs[0]].w[:4], l0.stride, l0.pad)
    rate = 4 * l0.ho * l0.wo * l0.k * l0.k * l0.cin / max(time.perf_counter() - t0, 1e-6)
    budget = min(1.0, 100.0 / max(1, args.steps + args.warmup))

    def sample(step):
        li = convs[step % len(convs)]
        l = wl.layers[li]
        per_ch = l.ho * l.wo * l.k * l.k * l.cin
        c_sub = int(np.clip(budget * rate * threads / per_ch, 1, l.cout))
        chunks = np.array_split(np.arange(c_sub), min(threads, c_sub))
        p, T, s = folded[li]

        def one(ch):
            sub = O.Params(p.alpha[ch], p.gamma[ch], p.beta[ch], p.mean[ch], p.var[ch], None, p.delta_in,
                           p.q_base, p.q_offset, p.eps, p.kbits)
            A = O.conv_acc(inputs[li], params[li].w[ch], l.stride, l.pad)
            O.check_chains(A, sub, T[ch], s[ch])

        with ThreadPoolExecutor(len(chunks)) as ex:
            list(ex.map(one, chunks))
        return 2.0 * per_ch * c_sub

    for i in range(args.warmup):
        sample(i)
    tot_ops, tot_t = 0.0, 0.0
    for i in range(args.steps):
        t0 = time.perf_counter()
        ops = sample(i)
        tot_t += time.perf_counter() - t0
        tot_ops += ops
    value = tot_ops / tot_t / 1e12
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot_t / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int32 (naive loops) + f64",
            "data": "synthetic", "config": line_config(wl, args),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                             "sample": f"each of {args.steps} steps: a slice of the output channels of one conv "
                                       f"layer for image 0 (cycling over {len(convs)} layers), both chains"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


POOL_HBM_SHAPE = (512, 208, 208, 32)   # Tiny-YOLO pool2 (2x2 / 2 on 208x208x32 codes) at batch 512


def measure_pool_hbm(ifq, torch, dev, stream, reps=20):
    """HBM throughput of the code max-pool (an HBM-bound step of the path) on a map larger than L2:
    2x2 / stride 2 on 512 x 208 x 208 x 32 packed 2-bit codes (177 MB in, 44 MB out), channel
    signs with negatives.  Launches back to back, each between CUDA events; the input is larger
    than L2 (129 MB), so no flush: a flush write would leave L2 full of dirty lines whose
    write-back the timed launch would pay for."""
    n, h, w, c = POOL_HBM_SHAPE
    d = ifq.pool_desc(n, h, w, c, 2, 2, 0, 2)
    ho, wo = ifq.ifq_pool_out_shape(d)
    g = torch.Generator(device=dev).manual_seed(1911_08076)
    x = torch.randint(0, 256, (n, h, w, c // 4), dtype=torch.uint8, device=dev, generator=g)
    y = torch.empty((n, ho, wo, c // 4), dtype=torch.uint8, device=dev)
    sign = torch.ones(c, dtype=torch.int8, device=dev)
    sign[1::3] = -1
    bytes_moved = x.numel() + y.numel()
    with torch.cuda.stream(stream):
        for _ in range(3):
            ifq.ifq_maxpool2bit(d, x, sign, y, stream)
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
        for a, b in ev:
            a.record(stream)
            ifq.ifq_maxpool2bit(d, x, sign, y, stream)
            b.record(stream)
        torch.cuda.synchronize()
    us = 1e3 * sum(a.elapsed_time(b) for a, b in ev) / reps
    _, _, hbm, src = read_peaks()
    gbs = bytes_moved / (us * 1e-6) / 1e9
    del x, y
    return {"kernel": "maxpool2x2_rowpair_kernel", "shape": f"2x2/2 pool, {n}x{h}x{w}x{c} 2-bit codes",
            "algorithmic_bytes": bytes_moved, "us": us, "achieved_gbs": gbs, "peak_gbs": hbm,
            "frac": gbs / hbm, "peak_source": f"{src} STREAM copy",
            "l2": "not flushed: input (177 MB) larger than L2 (129 MB)"}


def reduce_max(v: float, world: int, device) -> float:
    """The maximum of v over all ranks (the slowest replica sets the job's step time)."""
    if world == 1:
        return v
    import torch
    import torch.distributed as dist
    t = torch.tensor([v], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(ops_per_rank_step: float, world: int, step_ms_max: float) -> float:
    """Whole-job TOPS of `world` replicas, each doing ops_per_rank_step per step, at the max step time."""
    return world * ops_per_rank_step / (step_ms_max * 1e-3) / 1e12


PATH_NAMES = {0: "auto", 1: "conv_tc_kernel", 2: "bitserial", 3: "conv_direct_kernel", 4: "conv_win_kernel",
              5: "conv_warp_kernel"}


def kernel_of(ifq, st, li):
    """Name of the kernel family a layer launches (the planner's choice for convs)."""
    rec = st.layers[li]
    if rec.kind == ifq.IFQ_LAYER_CONV:
        p = ifq.ifq_conv_plan(rec.conv)
        if p == ifq.IFQ_PATH_BITSERIAL:
            l = st.wl.layers[li]
            narrow = l.kind == "conv" and l.cin in (4, 8, 16) and l.k == 3 and l.stride == 1 and l.cout <= 32
            return "conv_bitserial_narrow_kernel" if narrow else "conv_bitserial_kernel"
        return PATH_NAMES.get(p, str(p))
    if rec.kind == ifq.IFQ_LAYER_POOL:
        return "maxpool_codes"
    return "fixed_output_kernel"


def measure_workload(name, args, ifq, torch, dev, stream, flush, K, W, world, barrier, max_over_ranks,
                     peaks, e2e_separate=False, clocks=False):
    """Time one workload: K graph replays of the step (L2 flushed between steps, outside the
    step events), per-launch durations from a graph with external event nodes, the end-to-end
    step through ifq_graph_create_io from pinned host buffers, and the per-layer roofline.
    Returns (record, workload, inputs, params)."""
    from paper_1911_08076_gb300.stack import DeviceStack
    wl = synth.get(name, args.batch if name == args.workload else None)
    B = wl.batch
    x, params = synth.draw_workload(wl)
    path = {"auto": ifq.IFQ_PATH_AUTO, "tc": ifq.IFQ_PATH_TC, "bitserial": ifq.IFQ_PATH_BITSERIAL}[args.path]
    st = DeviceStack(wl, params, device=str(dev), path=path)
    x_host = torch.from_numpy(synth.pack_codes(x, 8 if wl.in_bits == 8 else wl.kbits)).pin_memory()
    xd = st.input_buffer()
    xd.copy_(x_host)
    torch.cuda.synchronize()
    st.capture(xd, stream)
    convs = [l for l in wl.layers if l.kind == "conv"]
    ops = sum(conv_ops(l, B) for l in convs)
    rec = {"workload": wl.name, "batch": B, "layers": len(wl.layers), "ops_per_step": ops}
    sampler = None
    with torch.cuda.stream(stream):
        for i in range(W):
            st.replay(stream)
            flush.fill_(i & 0xFF)
        torch.cuda.synchronize()
        starts = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
        ends = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
        if clocks:
            sampler = ClockSampler("GPU-" + str(torch.cuda.get_device_properties(dev).uuid))
            sampler.start()
        barrier()
        torch.cuda.synchronize()
        wall0 = time.perf_counter()
        for i in range(K):
            starts[i].record(stream)
            st.replay(stream)
            ends[i].record(stream)
            flush.fill_(i & 0xFF)
        torch.cuda.synchronize()
        wall = time.perf_counter() - wall0
        barrier()
        if sampler is not None:
            rec["clocks"] = sampler.stop()
        step_ms = max_over_ranks(sum(s.elapsed_time(e) for s, e in zip(starts, ends)) / K)
        status = ifq.ifq_device_status(stream)
        if status != ifq.IFQ_OK:
            raise RuntimeError(f"{wl.name}: device status after timed region: {ifq.ifq_status_str(status)}")

        # per-launch durations: the step's launches captured in a graph with an external event
        # record node around each kernel, replayed with an L2 flush before each step
        KR = max(3, min(K, 300))
        try:
            ev = [(torch.cuda.Event(enable_timing=True, external=True),
                   torch.cuda.Event(enable_timing=True, external=True)) for _ in wl.layers]
            g_ev = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g_ev, stream=stream):
                st.forward_layers(xd, before=lambda li: ev[li][0].record(stream),
                                  after=lambda li: ev[li][1].record(stream), stream=stream)
            timing_mode = "graph with external event nodes"
            acc = [0.0] * len(wl.layers)
            for i in range(KR):
                flush.fill_(i & 0xFF)
                g_ev.replay()
                torch.cuda.synchronize()
                for li in range(len(wl.layers)):
                    acc[li] += ev[li][0].elapsed_time(ev[li][1])
            per_layer_ms = [a / KR for a in acc]
            del g_ev
        except TypeError:
            # torch without external events: eager launches (includes host launch latency)
            timing_mode = "eager launches"
            evl = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                    for _ in wl.layers] for _ in range(KR)]
            for i in range(KR):
                flush.fill_(i & 0xFF)
                st.forward_layers(xd, before=lambda li, i=i: evl[i][li][0].record(stream),
                                  after=lambda li, i=i: evl[i][li][1].record(stream), stream=stream)
            torch.cuda.synchronize()
            per_layer_ms = [sum(evl[i][li][0].elapsed_time(evl[i][li][1]) for i in range(KR)) / KR
                            for li in range(len(wl.layers))]

        # end to end through the C ABI with host buffers: one graph launch per step that copies the
        # pinned host input in first and every result (the leaf layers' outputs) out right after its
        # layer (ifq_graph_create_io)
        leaf_host = torch.empty(st.leaf_block.shape, dtype=torch.uint8).pin_memory()
        h2d = x_host.numel() * x_host.element_size()
        d2h = sum(n for _, n in st.leaf_spans())
        KE = max(3, min(K, 1000))

        def timed_steps(step):
            for i in range(max(3, min(W, 20))):
                step()
            torch.cuda.synchronize()
            barrier()
            es = [torch.cuda.Event(enable_timing=True) for _ in range(KE)]
            ee = [torch.cuda.Event(enable_timing=True) for _ in range(KE)]
            for i in range(KE):
                es[i].record(stream)
                step()
                ee[i].record(stream)
                flush.fill_(i & 0xFF)
            torch.cuda.synchronize()
            return max_over_ranks(sum(s.elapsed_time(e) for s, e in zip(es, ee)) / KE)

        st.capture_io(xd, x_host, leaf_host, stream)
        e2e_ms = timed_steps(lambda: st.replay(stream))
        if not st.leaf_results_equal(leaf_host):
            raise RuntimeError(f"{wl.name}: end-to-end results differ from the device results")
        e2e = {"value": world * ops / (e2e_ms * 1e-3) / 1e12, "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms,
               "sequence": "per step (L2 flushed, untimed, between steps): one graph launch that copies the "
                           "pinned input in, runs the step and copies each result out after its layer"}
        if e2e_separate:
            st.capture(xd, stream)
            e2e_sep_ms = timed_steps(lambda: (ifq.ifq_copy_bytes(xd, x_host, h2d, stream), st.replay(stream),
                                              ifq.ifq_copy_bytes(leaf_host, st.leaf_block, leaf_host.numel(), stream)))
            e2e["separate_copies"] = {"value": world * ops / (e2e_sep_ms * 1e-3) / 1e12, "unit": UNIT,
                                      "ms_per_step": e2e_sep_ms,
                                      "sequence": "input copy, step graph, result copy: three launches"}

    # per-layer roofline: each launch timed alone against the tensor peak and the HBM copy rate
    peak, hbm = peaks["tensor_tops"], peaks["hbm_gbs"]
    layers = []
    for li, l in enumerate(wl.layers):
        us = 1e3 * per_layer_ms[li]
        b = layer_alg_bytes(wl, li, B)
        o = conv_ops(l, B) if l.kind == "conv" else 0.0
        t_tensor = o / (peak * 1e12) * 1e6
        t_hbm = b / (hbm * 1e9) * 1e6
        bound = "tensor" if t_tensor >= t_hbm else "hbm"
        layers.append({"name": l.name, "kernel": kernel_of(ifq, st, li), "us": round(us, 3),
                       "gop": round(o / 1e9, 4), "alg_mb": round(b / 1e6, 4),
                       "tops": round(o / (us * 1e-6) / 1e12, 2) if us > 0 else None,
                       "alg_gbs": round(b / (us * 1e-6) / 1e9, 1) if us > 0 else None,
                       "bound": bound, "roofline_us": round(max(t_tensor, t_hbm), 3),
                       "frac": round(max(t_tensor, t_hbm) / us, 4) if us > 0 else None})
    conv_idx = [i for i, l in enumerate(wl.layers) if l.kind == "conv"]
    conv_ms = sum(per_layer_ms[i] for i in conv_idx)
    total_ms = sum(per_layer_ms)
    conv_share = conv_ms / total_ms if total_ms > 0 else 1.0
    # A conv launch's in-step duration: the step's launches run back to back (programmatic dependent
    # launch overlaps each one's prologue with its predecessor's tail), so the convs' share of the
    # step time (from the serialised per-launch pass), divided by the conv launches per step.
    conv_in_step_ms = step_ms * conv_share
    achieved = ops / (conv_in_step_ms * 1e-3) / 1e12
    achieved_serial = ops / (conv_ms * 1e-3) / 1e12
    rec.update({
        "ms_per_step": step_ms, "value": job_throughput(ops, world, step_ms), "unit": UNIT,
        "images_per_s": world * B / (step_ms * 1e-3),
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak, "traffic": profiled_traffic(wl.name),
                     "kernel": "conv launches of a step" if len(conv_idx) > 1 else layers[conv_idx[0]]["kernel"],
                     "peak_source": peaks["tensor_source"],
                     "algorithmic_bytes_per_launch": sum(layer_alg_bytes(wl, i, B) for i in conv_idx) / len(conv_idx),
                     "ops_per_launch": ops / len(conv_idx),
                     "avg_launch_us": 1e3 * conv_in_step_ms / len(conv_idx),
                     "timing": "timed region: step time x conv share / conv launches per step",
                     "serialized": {"achieved": achieved_serial, "frac": achieved_serial / peak,
                                    "avg_launch_us": 1e3 * conv_ms / len(conv_idx),
                                    "timing": f"each launch alone between CUDA events ({timing_mode})"}},
        "e2e": e2e, "gpu_launches": K * len(wl.layers), "timed_wall_s": wall, "layers_timed_alone": layers,
    })
    log(f"{wl.name}: {step_ms * 1e3:.2f} us/step, {rec['value']:.1f} TOPS; per-layer us: " +
        ", ".join(f"{l['name']}={l['us']:.2f}" for l in layers))
    st.release()
    del st, xd
    torch.cuda.empty_cache()
    return rec, wl, x, params


def run_ours(args):
    import torch
    import torch.distributed as dist

    from paper_1911_08076_gb300 import ifq

    rank, world, local = dist_info()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)

    def barrier():
        if world > 1:
            dist.barrier()

    def max_over_ranks(v):
        return reduce_max(v, world, dev)

    stream = torch.cuda.Stream(device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    bf16, bf16_sus, hbm, src = read_peaks()
    peaks = {"tensor_tops": bf16 * FP8_PER_BF16, "hbm_gbs": hbm,
             "tensor_source": f"{src} bf16 burst {bf16} x {FP8_PER_BF16} (fp8/bf16 nominal)"}
    rates = measure_rates(stream)
    K, W = args.steps, args.warmup

    head, wl, x, params = measure_workload(args.workload, args, ifq, torch, dev, stream, flush, K, W, world,
                                           barrier, max_over_ranks, peaks, e2e_separate=True, clocks=True)
    value = head["value"]
    r = head["roofline"]
    ach = r["achieved"]

    def frac(v):
        return ach / v if v else None

    r["vs_measured_rates"] = {
        "tcgen05_e4m3_n128": frac(rates.get("tcgen05_e4m3_n128_tops")),
        "tcgen05_e4m3_n256": frac(rates.get("tcgen05_e4m3_n256_tops")),
        "tcgen05_e4m3_tmem_a_n128": frac(rates.get("tcgen05_e4m3_tmem_a_n128_tops")),
        "note": "achieved / the e4m3 tcgen05 rate measured in this process (the conv's own instruction; "
                "tmem_a: with A in tensor memory, the operand form the conv issues)"}
    s8 = rates.get("mma_sync_s8_tops")
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K, "warmup": W,
        "ms_per_step": head["ms_per_step"], "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": f"e4m3xe4m3->f32 (exact integer: u{wl.kbits} codes x +-1 signs)", "data": "synthetic",
        "config": line_config(wl, args),
        "images_per_s": head["images_per_s"],
        "pct_of_int8_peak": 100.0 * value / (world * s8) if s8 else None,
        "int8_peak": {"tops": s8, "source": "mma.sync.m16n8k32 s8 rate measured in this process (sm_103a has no "
                                            "tcgen05 integer MMA; the exact binary x 2-bit product runs on e4m3)"},
        "rates_measured": rates,
        "roofline": r,
        "e2e": head["e2e"],
        "gpu_launches": head["gpu_launches"],
        "clocks": head.get("clocks"),
        "timed_wall_s": head["timed_wall_s"],
        "layers_timed_alone": head["layers_timed_alone"],
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(wl, x, params, 12.0)
    del x, params
    subs = {}
    if not args.no_sub:
        for name in SUB_WORKLOADS:
            if name == args.workload:
                continue
            rec, swl, sx, sp = measure_workload(name, args, ifq, torch, dev, stream, flush, K, W, world, barrier,
                                                max_over_ranks, peaks)
            if rank == 0 and world == 1 and not args.no_cpu_baseline:
                rec["cpu_baseline"] = cpu_baseline(swl, sx, sp, 3.0)
            subs[name] = rec
    line["configs"] = subs
    line["pool_hbm"] = measure_pool_hbm(ifq, torch, dev, stream)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=HEADLINE, choices=sorted(synth.WORKLOADS))
    ap.add_argument("--batch", type=int, default=None)
    ap.add_argument("--path", default="auto", choices=["auto", "tc", "bitserial"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-sub", action="store_true", help="time the headline workload only")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
