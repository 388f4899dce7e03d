"""Benchmark of the quantized HWC convolution hot path on GB300.

Workload (one "step"): the paper's benchmark layer (Sec. V-A: 16x16x32 HWC
input, 64 filters 3x3x32, stride 1, pad 1) at batch 512, INT-8, compression
with per-channel kappa/lambda and shift 12: one qconv_hwc_run call on filters
prepared once with qconv_hwc_prepare when the layer is set up (the filters of
an inference layer are constants, as in the paper, where they sit in memory
already in the kernel's HWC order).  The one-shot qconv_hwc call, which
prepares the filters inside the same launch, is timed beside it and reported
as "oneshot".  Metric: GMAC/s.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Timing: W eager warm-up steps, then runs of exactly K steps replayed from CUDA
graphs, back to back, each run timed with its own CUDA events on the launching
stream, until at least 50 runs and one second are timed; the median run counts.
All runs are bracketed by a barrier and torch.cuda.synchronize() on both sides;
max over ranks.  Each step reads and
writes its own buffer set, rotating over sets whose total exceeds the 129 MB
L2, so every step streams its activations from HBM.

--impl reference times the oracle (the plain CPU implementation of the same
layer) on the host cores, on bounded samples of the same workload.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_1908_11263_gb300 import inputs  # noqa: E402

L2_BYTES = 129 * 1024 * 1024
# timed runs of the k-step graph: at least this many, and at least this long in all
MIN_REPLAYS, MIN_TIMED_SECONDS, MAX_REPLAYS = 50, 1.0, 20000
# nominal dense-rate ratio of e4m3 (kind::f8f6f4) to fp16 (kind::f16) tensor-core MMAs;
# only the bf16 rate is measured, so the e4m3 roof is that rate scaled by this ratio
E4M3_PER_FP16 = 2.0
WORKLOAD = "conv3x3_16x16x32_to_64_int8_n512"
INT8_IMMA_TOPS = 151.6
# 32-bit population counts per second on this GPU (all SMs; measured, 15.1 per SM per cycle at
# 2070 MHz): the ALU roof of the INT-1 convolution, 32 binary MACs per count
POPC_TPS = 4.77
METRIC = "qconv_hwc GMAC/s (16x16x32 -> 64, 3x3, stride 1, pad 1, INT-8, batch 512)"


PROFILE = os.path.join(ROOT, "profiles", "conv_win_kernel_conv3x3_16x16x32to64_int8_n512.md")
KERNEL_SOURCES = ("conv_win.cuh", "conv_win_inst.cuh", "conv_common.cuh", "device.cuh", "internal.h")
KERNEL_NAME = "conv_win_kernel<8,64,false,false>"


def measured_traffic():
    """DRAM bytes per launch of the timed convolution kernel, from the committed
    ncu summary, or None when the kernel's sources changed since that capture."""
    import hashlib
    try:
        line = next(l for l in open(PROFILE) if l.startswith("traffic:"))
        rec = json.loads(line[len("traffic:"):])
    except (OSError, StopIteration, ValueError):
        return None
    h = hashlib.sha256()
    for f in KERNEL_SOURCES:
        with open(os.path.join(ROOT, "paper_1908_11263_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return rec["dram_bytes_per_launch"] if h.hexdigest() == rec["source_sha256"] else None


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return dict(hbm_gbs=p["hbm_gbs"], bf16_tflops=p["bf16_tflops"], source="measured")
    return dict(hbm_gbs=6800.0, bf16_tflops=1900.0, source="fallback")


# ---------------------------------------------------------------------------- distributed plumbing

def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        import torch
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend=backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(value: float, world: int, device=None) -> float:
    """Largest value over all ranks (the slowest rank sets the whole-job time)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank_step: float, world: int, steps: int, t_max: float) -> float:
    """Units every rank processed, per second of the slowest rank's time (weak
    scaling: each rank runs `steps` steps of the same size on its own shard)."""
    return world * units_per_rank_step * steps / t_max


# ---------------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu):
        self.gpu = gpu
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if self.proc is None or not self.path or not os.path.exists(self.path):
            return None
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        smax = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower().startswith("active")})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": reasons, "samples": len(rows)}


# ---------------------------------------------------------------------------- our arm

def run_ours(args, world, rank, local):
    import torch
    from paper_1908_11263_gb300 import qnn

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    qnn.load(build_if_missing=True)
    (key, layer, wl, lid), = inputs.single_layer_workload(inputs.WORKLOAD_BATCH)
    ld = inputs.make_layer(key, layer, wl, lid)
    macs = layer.macs
    x0 = torch.from_numpy(ld.x).to(dev)
    w = torch.from_numpy(ld.w).to(dev)
    kappa = torch.from_numpy(ld.kappa).to(dev)
    lam = torch.from_numpy(ld.lam).to(dev)
    bias = torch.from_numpy(ld.bias).to(dev)
    per_set = x0.numel() + layer.n * layer.oh * layer.ow * layer.m
    nsets = max(2, math.ceil(2 * L2_BYTES / per_set))
    xs = [x0.clone() for _ in range(nsets)]
    ys = [torch.empty((layer.n, layer.oh, layer.ow, layer.m), dtype=torch.uint8, device=dev) for _ in range(nsets)]
    desc = qnn.conv_desc(layer.n, layer.h, layer.w, layer.c, layer.m, layer.k, layer.k, layer.stride, layer.pad, 8,
                         ld.shift)
    assert qnn.tc_kernel(desc) == qnn.ALGO_TC_WINDOW
    ws = torch.empty(qnn.workspace_size(desc), dtype=torch.uint8, device=dev)
    stream = torch.cuda.Stream(device=dev)
    launches_per_step = 1  # the window kernel: filter re-layout, convolution and compression in one launch

    prepared = qnn.PreparedConv(w, kappa, lam, n=layer.n, h=layer.h, wd=layer.w, bias=bias, shift=ld.shift, bits=8,
                                stride=1, pad=1, stream=stream)

    def step(i):  # one launch: the convolution on the prepared filters
        prepared(xs[i % nsets], out=ys[i % nsets], stream=stream)

    def oneshot(i):  # one launch that also prepares the filters from the caller's buffers
        qnn.conv_hwc(xs[i % nsets], w, kappa, lam, bias=bias, shift=ld.shift, bits=8, stride=1, pad=1,
                     out=ys[i % nsets], workspace=ws, stream=stream)

    warmup = max(3, args.warmup)
    with torch.cuda.stream(stream):
        for i in range(warmup):
            step(i)
            oneshot(i)
    qnn.device_status(stream)

    def capture(fn, count, offset, bulk=False):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            if bulk:
                fn(offset, count)
            else:
                for i in range(count):
                    fn(offset + i)
        return g

    def timed(fn, k, bulk=False, min_reps=MIN_REPLAYS, min_seconds=MIN_TIMED_SECONDS):
        """Median time of one run of exactly k steps.  The k steps are captured once
        (graphs of at most 1000 steps) and the whole k-step run is replayed back to
        back, each run bracketed by its own pair of CUDA events on the launching
        stream, until at least min_reps runs and min_seconds have been timed; the
        median run is returned (seconds) with the number of runs."""
        chunk = min(k, 1000)
        full, rem = divmod(k, chunk)
        g_full = capture(fn, chunk, 0, bulk)
        g_rem = capture(fn, rem, chunk, bulk) if rem else None

        def run():
            for _ in range(full):
                g_full.replay()
            if g_rem is not None:
                g_rem.replay()

        run()  # settle
        torch.cuda.synchronize(dev)
        # a first timed run sizes the repetition count
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record(stream)
            run()
            e1.record(stream)
        torch.cuda.synchronize(dev)
        one = max(e0.elapsed_time(e1) / 1e3, 1e-7)
        reps = int(min(MAX_REPLAYS, max(min_reps, math.ceil(min_seconds / one))))
        events = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
        barrier(world)
        torch.cuda.synchronize(dev)
        with torch.cuda.stream(stream):
            for a, b in events:
                a.record(stream)
                run()
                b.record(stream)
        torch.cuda.synchronize(dev)
        barrier(world)
        times = [a.elapsed_time(b) / 1e3 for a, b in events]
        return statistics.median(times), reps

    k = args.steps
    try:
        gpu_id = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        gpu_id = str(local)
    with ClockSampler(gpu_id) as clk:
        t_step, reps = timed(step, k)
        t_oneshot, _ = timed(oneshot, k)
    qnn.device_status(stream)
    t_max = max_over_ranks(t_step, world, dev)
    clocks = clk.summary()

    # End to end through the public API with host buffers: every step copies its input
    # from pinned host memory, runs qconv_hwc and copies its output back to pinned host
    # memory.  Consecutive steps stream through three CUDA streams (input copies,
    # compute, output copies) ordered by events, so the copies of one step overlap
    # the compute of its neighbours; rotating device buffers carry the WAR ordering.
    xh = torch.from_numpy(ld.x).pin_memory()
    yh = torch.empty(ys[0].shape, dtype=torch.uint8).pin_memory()
    s_in, s_out = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    ring = nsets + 2
    ev_in = [torch.cuda.Event() for _ in range(ring)]
    ev_c = [torch.cuda.Event() for _ in range(ring)]
    ev_out = [torch.cuda.Event() for _ in range(ring)]

    def e2e_steps(offset, count):
        fork = torch.cuda.Event()
        fork.record(stream)
        s_in.wait_event(fork)
        s_out.wait_event(fork)
        for j in range(count):
            i = offset + j
            if j >= nsets:
                s_in.wait_event(ev_c[(j - nsets) % ring])  # compute of the set's previous step has read it
            with torch.cuda.stream(s_in):
                xs[i % nsets].copy_(xh, non_blocking=True)
            ev_in[j % ring].record(s_in)
            stream.wait_event(ev_in[j % ring])
            if j >= nsets:
                stream.wait_event(ev_out[(j - nsets) % ring])  # output copy of the set's previous step is done
            step(i)
            ev_c[j % ring].record(stream)
            s_out.wait_event(ev_c[j % ring])
            with torch.cuda.stream(s_out):
                yh.copy_(ys[i % nsets], non_blocking=True)
            ev_out[j % ring].record(s_out)
        for s_side in (s_in, s_out):  # join
            ev = torch.cuda.Event()
            ev.record(s_side)
            stream.wait_event(ev)

    with torch.cuda.stream(stream):
        e2e_steps(0, 3)
    e2e_k = max(10, min(k, 2000))
    t_e2e = max_over_ranks(timed(e2e_steps, e2e_k, bulk=True, min_reps=5, min_seconds=0.05)[0], world, dev)

    # parity spot-check of the last output set against a second, independent GPU kernel
    ref = qnn.conv_hwc(xs[0], w, kappa, lam, bias=bias, shift=ld.shift, bits=8, stride=1, pad=1,
                       algo=qnn.ALGO_DIRECT)
    torch.cuda.synchronize(dev)
    if not torch.equal(ref, ys[0]):
        raise SystemExit("bench: tensor-core output differs from the CUDA-core kernel")

    pk = peaks()
    flops = 2.0 * macs
    kernel_s = t_step / k  # one kernel launch per step
    achieved_tflops = flops / kernel_s / 1e12
    alg_bytes = layer.algorithmic_bytes()
    result = None
    if rank == 0:
        gmacs = whole_job_rate(macs, world, k, t_max) / 1e9
        result = {
            "metric": METRIC,
            "value": round(gmacs, 1),
            "unit": "GMAC/s",
            "n_gpus": world,
            "steps": k,
            "warmup": warmup,
            "ms_per_step": round(t_max / k * 1e3, 6),
            "higher_is_better": True,
            "scaling": "weak",
            "vs_baseline": None,
            "dtype": "u8*s8->i32 (exact fp16 tensor-core embedding)",
            "data": "synthetic (seeded SplitMix64, uniform INT-8 values; same shapes as the paper's layer)",
            "config": {"workload": WORKLOAD, "batch": layer.n, "input_hwc": [layer.h, layer.w, layer.c],
                       "filters": [layer.m, layer.k, layer.k, layer.c], "stride": 1, "pad": 1, "bits": 8,
                       "shift": ld.shift, "parallelism": f"replicas x{world}",
                       "l2": f"rotating {nsets} buffer sets ({nsets * per_set / 2**20:.0f} MiB > L2)",
                       "timing": f"median of {reps} back-to-back runs of exactly {k} steps (CUDA graphs of "
                                 f"qconv_hwc_run calls on prepared filters), each run timed with CUDA events on the launching stream"},
            "gpu_launches": launches_per_step * k,
            "roofline": {
                "kernel": KERNEL_NAME,
                "bound": "tensor",
                "achieved": round(achieved_tflops, 1),
                "peak": pk["bf16_tflops"],
                "unit": "TFLOP/s",
                "frac": round(achieved_tflops / pk["bf16_tflops"], 4),
                "peak_source": f"{pk['source']} bf16 dense burst (fp16 has the same nominal rate)",
                "kernel_us": round(kernel_s * 1e6, 3),
                "algorithmic_flops": flops,
                "algorithmic_bytes": alg_bytes,
                "hbm_frac_at_this_time": round(alg_bytes / kernel_s / 1e9 / pk["hbm_gbs"], 4),
                "traffic": measured_traffic(),
            },
            # the only INT8 tensor path on sm_103a is the warp-level mma.sync IMMA (no tcgen05 kind::i8);
            # its rate on this GPU, measured with m16n8k32 u8*s8 MMAs from all SMs, is context only
            "int8_tensor_ref": {"peak_tops": INT8_IMMA_TOPS, "frac": round(achieved_tflops / INT8_IMMA_TOPS, 3),
                                "source": "measured mma.sync.m16n8k32 u8*s8 rate, all SMs, GB300"},
            "e2e": {"value": round(whole_job_rate(macs, world, e2e_k, t_e2e) / 1e9, 1), "unit": "GMAC/s",
                    "h2d_bytes_per_step": int(xh.numel()), "d2h_bytes_per_step": int(yh.numel()),
                    "steps": e2e_k,
                    "pipeline": "input copy, compute and output copy of consecutive steps on three streams"},
            "clocks": clocks,
            "oneshot": {"value": round(whole_job_rate(macs, world, k, t_oneshot) / 1e9, 1), "unit": "GMAC/s",
                        "us_per_step": round(t_oneshot / k * 1e6, 3),
                        "what": "qconv_hwc with the caller's raw filters: the same kernel, preparing the filters "
                                "inside the launch (no workspace)"},
        }
        if clocks and clocks.get("sm_mhz"):
            # clock-normalised step time: compare runs taken at different SM clocks
            clocks["step_us_x_sm_mhz"] = round(t_max / k * 1e6 * clocks["sm_mhz"], 1)
        if args.cpu_baseline:
            result["cpu_baseline"] = oracle_baseline(layer, ld, budget_s=args.cpu_seconds)
    return result


# ---------------------------------------------------------------------------- the oracle on host cores

def oracle_sample_rate(layer, ld, nimg, threads):
    import oracle
    shape = layer.shape()
    shape["n"] = nimg
    xs = ld.x[:nimg].reshape(-1)
    ws = ld.w.reshape(-1).view(np.uint8)
    t0 = time.perf_counter()
    oracle.conv_hwc(xs, ws, shape, ld.bias, ld.kappa, ld.lam, shift=ld.shift, nthreads=threads)
    dt = time.perf_counter() - t0
    return dt, nimg * layer.macs / layer.n


def oracle_baseline(layer, ld, budget_s=15.0):
    """The oracle as it stands, on all host cores, on a bounded sample of about budget_s seconds:
    a batch prefix of the workload, or, when the whole batch takes less than half the budget,
    the whole batch repeated to fill it."""
    threads = os.cpu_count() or 1
    probe = max(1, min(layer.n, threads))
    dt, macs = oracle_sample_rate(layer, ld, probe, threads)
    nimg = int(min(layer.n, max(probe, probe * budget_s / max(dt, 1e-6))))
    dt, macs = oracle_sample_rate(layer, ld, nimg, threads)
    passes = 1
    if nimg == layer.n and dt < budget_s / 2:
        passes = max(1, int(budget_s / max(dt, 1e-6)))
        dt, macs = 0.0, 0.0
        for _ in range(passes):
            d, m = oracle_sample_rate(layer, ld, nimg, threads)
            dt += d
            macs += m
    return {"value": round(macs / dt / 1e9, 3), "unit": "GMAC/s", "cores": threads, "kind": "oracle",
            "sample": f"{nimg} of {layer.n} images of the workload x {passes} pass{'es' if passes > 1 else ''} "
                      f"({macs / 1e9:.2f} GMAC, {dt:.1f} s, OpenMP over images)"}


def run_reference(args, world, rank):
    if rank != 0:
        return None
    (key, layer, wl, lid), = inputs.single_layer_workload(inputs.WORKLOAD_BATCH)
    ld = inputs.make_layer(key, layer, wl, lid)
    threads = os.cpu_count() or 1
    steps, warmup = args.steps, max(0, args.warmup)
    # size each step so the whole run stays within about two minutes
    dt1, _ = oracle_sample_rate(layer, ld, max(1, threads), threads)
    per_img = dt1 / max(1, threads)
    budget = min(2.0, 120.0 / max(1, steps + warmup))
    nimg = int(max(1, min(layer.n, budget / max(per_img, 1e-9))))
    for _ in range(warmup):
        oracle_sample_rate(layer, ld, nimg, threads)
    times = []
    macs = 0
    for _ in range(steps):
        dt, macs = oracle_sample_rate(layer, ld, nimg, threads)
        times.append(dt)
    total = sum(times)
    value = steps * macs / total / 1e9
    sample = f"{nimg} of {layer.n} images per step ({macs / 1e9:.3f} GMAC), OpenMP over images"
    return {
        "impl": "reference",
        "metric": METRIC,
        "value": round(value, 3),
        "unit": "GMAC/s",
        "n_gpus": world,
        "steps": steps,
        "warmup": warmup,
        "ms_per_step": round(total / steps * 1e3, 3),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "int64 (plain C oracle)",
        "data": "synthetic (seeded SplitMix64, uniform INT-8 values; same shapes as the paper's layer)",
        "config": {"workload": WORKLOAD, "batch": layer.n, "sample_images_per_step": nimg},
        "cpu_baseline": {"value": round(value, 3), "unit": "GMAC/s", "cores": threads, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": round(value, 3), "unit": "GMAC/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


# ---------------------------------------------------------------------------- per-config sweep

def run_sweep(args):
    """One JSON line per layer of workloads 1 to 5:
    GMAC/s of qconv_hwc calls and of the convolution kernel alone, each timed from CUDA
    graphs over rotating buffer sets larger than L2, with the roof that binds the layer
    (its arithmetic intensity against the measured ridge) and the fraction reached."""
    import torch
    from paper_1908_11263_gb300 import qnn
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    qnn.load(build_if_missing=True)
    pk = peaks()
    stream = torch.cuda.Stream(device=dev)

    def dev_packed(vals, bits, shape_bytes):
        t = torch.from_numpy(np.ascontiguousarray(vals).reshape(-1).astype(np.int8)).to(dev)
        if bits != 8:
            t = qnn.pack_subbyte(t, bits, stream=stream)
        return t.view(torch.uint8).view(shape_bytes)

    def graph_time(fn, count, reps):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for i in range(count):
                fn(i)
        g.replay()
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record(stream)
            for _ in range(reps):
                g.replay()
            e1.record(stream)
        torch.cuda.synchronize(dev)
        return e0.elapsed_time(e1) / 1e3 / (count * reps)

    def layer_tensors(key, layer, wl, lid, with_x=True):
        # without an input of its own (pipeline layers) the layer's input is not drawn
        ld = inputs.make_layer(key, layer, wl, lid, x=None if with_x else np.zeros(1, np.int64))
        per = 8 // layer.bits
        t = dict(
            w=dev_packed(ld.w, layer.bits, (layer.m, layer.k, layer.k, layer.c // per)),
            kappa=torch.from_numpy(ld.kappa).to(dev), lam=torch.from_numpy(ld.lam).to(dev),
            bias=torch.from_numpy(ld.bias).to(dev),
            shifts=None if ld.shifts is None else torch.from_numpy(ld.shifts).to(dev), shift=ld.shift)
        if with_x:
            t["x"] = dev_packed(ld.x, layer.bits, (layer.n, layer.h, layer.w, layer.c // per))
        return ld, t

    def roof(flops, nbytes, seconds, operand_bits=16):
        """The binding roof of a layer: tensor when its arithmetic intensity exceeds the ridge
        of the tensor rate its MMAs run at (fp16, or e4m3 at the nominal 2x the measured
        bf16/fp16 rate), else HBM."""
        scale = E4M3_PER_FP16 if operand_bits == 8 else 1.0
        tpeak = pk["bf16_tflops"] * scale
        ai = flops / nbytes
        if ai >= tpeak * 1e12 / (pk["hbm_gbs"] * 1e9):
            src = (f"{pk['source']} bf16 dense burst x {E4M3_PER_FP16:g} (nominal e4m3:fp16 rate ratio; "
                   f"kind::f8f6f4 MMAs)" if operand_bits == 8 else
                   f"{pk['source']} bf16 dense burst (fp16 kind::f16 MMAs, same nominal rate)")
            return {"bound": "tensor", "achieved": round(flops / seconds / 1e12, 1), "peak": round(tpeak, 1),
                    "unit": "TFLOP/s", "frac": round(flops / seconds / 1e12 / tpeak, 4),
                    "arith_intensity": round(ai, 1), "peak_source": src}
        return {"bound": "hbm", "achieved": round(nbytes / seconds / 1e9, 1), "peak": pk["hbm_gbs"], "unit": "GB/s",
                "frac": round(nbytes / seconds / 1e9 / pk["hbm_gbs"], 4), "arith_intensity": round(ai, 1),
                "peak_source": f"{pk['source']} HBM copy bandwidth"}

    def oracle_times(layer, ld):
        """The oracle on this layer: one thread on a batch prefix of about 1.5 s, scaled to the
        whole batch, and all host cores on the whole batch (OpenMP over images)."""
        import oracle
        if not args.oracle_times:
            return None
        per = 8 // layer.bits
        xs = ld.x.reshape(layer.n, -1)
        wp = ld.w.reshape(-1).astype(np.int8).view(np.uint8) if layer.bits == 8 else oracle.pack(ld.w.reshape(-1), layer.bits)
        threads = os.cpu_count() or 1

        def run(nimg, nth):
            shape = layer.shape()
            shape["n"] = nimg
            xi = xs[:nimg].reshape(-1)
            xp = xi.astype(np.uint8) if layer.bits == 8 else oracle.pack(xi, layer.bits)
            t0 = time.perf_counter()
            oracle.conv_hwc(xp, wp, shape, ld.bias, ld.kappa, ld.lam, shifts=ld.shifts, shift=ld.shift, nthreads=nth)
            return time.perf_counter() - t0

        t1 = run(1, 1)
        n1 = int(max(1, min(layer.n, 1.5 / max(t1, 1e-6))))
        t1 = run(n1, 1) * layer.n / n1
        tall = run(layer.n, threads)
        return {"one_thread_s": round(t1, 4), "one_thread_sample": f"{n1} of {layer.n} images, scaled",
                "all_cores_s": round(tall, 4), "cores": threads, "per_image_bytes": layer.h * layer.w * layer.c // per}

    def conv_line(config, key, layer, wl, lid, extra=None):
        ld, t = layer_tensors(key, layer, wl, lid)
        per = 8 // layer.bits
        set_bytes = t["x"].numel() + layer.n * layer.oh * layer.ow * layer.m // per
        nsets = max(2, math.ceil(2 * L2_BYTES / set_bytes))
        xs = [t["x"].clone() for _ in range(nsets)]
        ys = [torch.empty((layer.n, layer.oh, layer.ow, layer.m // per), dtype=torch.uint8, device=dev)
              for _ in range(nsets)]
        kw = dict(bias=t["bias"], shifts=t["shifts"], shift=t["shift"], bits=layer.bits, stride=layer.stride,
                  pad=layer.pad)
        desc = qnn.conv_desc(layer.n, layer.h, layer.w, layer.c, layer.m, layer.k, layer.k, layer.stride,
                             layer.pad, layer.bits, t["shift"])
        algo = qnn.conv_algo(desc)
        ws = torch.empty(max(1, qnn.workspace_size(desc)), dtype=torch.uint8, device=dev)

        def call(i):
            qnn.conv_hwc(xs[i % nsets], t["w"], t["kappa"], t["lam"], out=ys[i % nsets], workspace=ws,
                         stream=stream, **kw)

        with torch.cuda.stream(stream):
            for i in range(3):
                call(i)
        torch.cuda.synchronize(dev)
        count = max(20, min(1000, int(2e9 / max(layer.macs, 1))))
        t_call = graph_time(call, count, 3)
        t_kernel = None
        if algo == qnn.ALGO_TENSORCORE:
            prepared = qnn.PreparedConv(t["w"], t["kappa"], t["lam"], n=layer.n, h=layer.h, wd=layer.w,
                                        bias=t["bias"], shifts=t["shifts"], shift=t["shift"], bits=layer.bits,
                                        stride=layer.stride, pad=layer.pad, stream=stream)
            t_kernel = graph_time(lambda i: prepared(xs[i % nsets], out=ys[i % nsets], stream=stream), count, 3)
        qnn.device_status(stream)
        tk = t_kernel if t_kernel is not None else t_call
        opbits = qnn.mma_operand_bits(desc)
        kernel = {qnn.ALGO_TC_WINDOW: "window", qnn.ALGO_TC_GENERAL: "general", 0: "direct"}[qnn.tc_kernel(desc)]
        line = {"sweep": config, "layer": layer.name, "algo": "tensorcore" if algo == qnn.ALGO_TENSORCORE else "direct",
                "kernel": kernel,
                "mma_operands": {16: "fp16", 8: "e4m3", 0: "none (CUDA cores)"}[opbits],
                "macs": layer.macs, "gmacs_call": round(layer.macs / t_call / 1e9, 1), "us_call": round(t_call * 1e6, 3),
                "gmacs_kernel": round(layer.macs / tk / 1e9, 1), "us_kernel": round(tk * 1e6, 3),
                "algorithmic_bytes": layer.algorithmic_bytes(),
                "roofline": roof(2.0 * layer.macs, layer.algorithmic_bytes(), tk, opbits),
                "oracle": oracle_times(layer, ld), "l2": f"rotating {nsets} buffer sets"}
        if extra:
            line.update(extra)
        print(json.dumps(line), flush=True)
        return t_call

    # config 1: batch 1, latency; graph-captured and plain launches
    (key, layer, wl, lid), = inputs.single_layer_workload(inputs.WORKLOAD_SINGLE)
    t_graph = conv_line("1", key, layer, wl, lid)
    ld, t = layer_tensors(key, layer, wl, lid)
    y = torch.empty((1, 16, 16, 64), dtype=torch.uint8, device=dev)
    with torch.cuda.stream(stream):
        for _ in range(20):
            qnn.conv_hwc(t["x"], t["w"], t["kappa"], t["lam"], bias=t["bias"], shift=t["shift"], pad=1, out=y,
                         stream=stream)
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(200):
            qnn.conv_hwc(t["x"], t["w"], t["kappa"], t["lam"], bias=t["bias"], shift=t["shift"], pad=1, out=y,
                         stream=stream)
        e1.record(stream)
    torch.cuda.synchronize(dev)
    t_plain = e0.elapsed_time(e1) / 1e3 / 200
    print(json.dumps({"sweep": "1", "layer": layer.name, "us_call_graph": round(t_graph * 1e6, 3),
                      "us_call_plain_launch": round(t_plain * 1e6, 3)}), flush=True)

    # config 2: the default run's layer, here with the same per-layer columns as the others
    (key, layer, wl, lid), = inputs.single_layer_workload(inputs.WORKLOAD_BATCH)
    conv_line("2", key, layer, wl, lid)
    # config 4: INT-4 and INT-2
    for key, layer, wl, lid in inputs.single_layer_workload(inputs.WORKLOAD_SUBBYTE):
        conv_line("4", key, layer, wl, lid)
    # config 5: larger layers at batch 64
    for key, layer, wl, lid in inputs.single_layer_workload(inputs.WORKLOAD_SWEEP):
        conv_line("5", key, layer, wl, lid)
    # config 3: the CIFAR-shaped network, each layer, then the whole pipeline
    layers = inputs.cifar_layers(1024)
    for key, layer, wl, lid in layers:
        conv_line("3", key, layer, wl, lid)
    run_cifar_pipeline(layers, layer_tensors, graph_time, stream, dev)
    run_pool_linear(graph_time, stream, dev, pk)
    run_binary(graph_time, stream, dev)


def run_binary(graph_time, stream, dev):
    """INT-1 (XNOR / popcount) convolution on the benchmark layer's shape, against the popcount roof."""
    import torch
    from paper_1908_11263_gb300 import qnn
    rng = np.random.default_rng(12)
    n, h, w, c, m, k = 512, 16, 16, 32, 64, 3
    xbytes, ybytes = n * h * w * c // 8, n * h * w * m // 8
    nsets = max(2, math.ceil(2 * L2_BYTES / (xbytes + ybytes)))
    xs = [torch.from_numpy(rng.integers(0, 256, size=(n, h, w, c // 8), dtype=np.uint8)).to(dev) for _ in range(nsets)]
    wt = torch.from_numpy(rng.integers(0, 256, size=(m, k, k, c // 8), dtype=np.uint8)).to(dev)
    tau = torch.full((m,), k * k * c // 2, dtype=torch.int32, device=dev)
    ys = [torch.empty((n, h, w, m // 8), dtype=torch.uint8, device=dev) for _ in range(nsets)]
    t = graph_time(lambda i: qnn.conv_binary(xs[i % nsets], wt, tau, pad=1, out=ys[i % nsets], stream=stream), 200, 3)
    qnn.device_status(stream)
    macs = n * h * w * m * k * k * c
    achieved = macs / t / 1e12
    peak = POPC_TPS * 32
    print(json.dumps({"sweep": "int1", "layer": "binary conv3x3_16x16x32_to_64 n512 (XNOR/popcount)",
                      "macs": macs, "us_kernel": round(t * 1e6, 3), "gmacs_kernel": round(macs / t / 1e9, 1),
                      "roofline": {"bound": "alu", "achieved": round(achieved, 2), "peak": round(peak, 1),
                                   "unit": "T binary MAC/s", "frac": round(achieved / peak, 4),
                                   "peak_source": "measured popc rate x 32 bits per count"},
                      "l2": f"rotating {nsets} buffer sets"}), flush=True)


def run_pool_linear(graph_time, stream, dev, pk):
    """qmaxpool (2x2, stride 2) and qlinear on the CIFAR network's shapes, against the HBM roof."""
    import torch
    from paper_1908_11263_gb300 import qnn
    rng = np.random.default_rng(11)
    for (n, h, w, c, bits) in ((1024, 32, 32, 32, 8), (1024, 16, 16, 32, 8), (1024, 8, 8, 64, 8),
                               (512, 16, 16, 64, 4), (512, 16, 16, 64, 2)):
        per = 8 // bits
        in_bytes = n * h * w * c // per
        out_bytes = in_bytes // 4
        nsets = max(2, math.ceil(2 * L2_BYTES / (in_bytes + out_bytes)))
        xs = [torch.from_numpy(rng.integers(0, 256, size=(n, h, w, c // per), dtype=np.uint8)).to(dev)
              for _ in range(min(nsets, 4))]
        xs = [xs[i % len(xs)].clone() for i in range(nsets)]
        ys = [torch.empty((n, h // 2, w // 2, c // per), dtype=torch.uint8, device=dev) for _ in range(nsets)]
        t = graph_time(lambda i: qnn.maxpool(xs[i % nsets], 2, 2, bits, out=ys[i % nsets], stream=stream), 200, 3)
        gbs = (in_bytes + out_bytes) / t / 1e9
        print(json.dumps({"sweep": "pool", "layer": f"qmaxpool 2x2/2 {n}x{h}x{w}x{c} INT-{bits}",
                          "us_kernel": round(t * 1e6, 3), "algorithmic_bytes": in_bytes + out_bytes,
                          "roofline": {"bound": "hbm", "achieved": round(gbs, 1), "peak": pk["hbm_gbs"],
                                       "unit": "GB/s", "frac": round(gbs / pk["hbm_gbs"], 4)},
                          "l2": f"rotating {nsets} buffer sets"}), flush=True)
    n, k, m = 1024, 1024, 10
    nsets = max(2, math.ceil(2 * L2_BYTES / (n * k + n * m * 4)))
    xs = [torch.from_numpy(rng.integers(0, 256, size=(n, k), dtype=np.uint8)).to(dev) for _ in range(nsets)]
    wt = torch.from_numpy(rng.integers(-128, 128, size=(m, k), dtype=np.int8)).to(dev)
    bias = torch.from_numpy(rng.integers(-4096, 4097, size=m).astype(np.int32)).to(dev)
    ys = [torch.empty((n, m), dtype=torch.int32, device=dev) for _ in range(nsets)]
    t = graph_time(lambda i: qnn.linear(xs[i % nsets], wt, bias, out=ys[i % nsets], stream=stream), 200, 3)
    nbytes = n * k + m * k + m * 4 + n * m * 4
    gbs = nbytes / t / 1e9
    print(json.dumps({"sweep": "linear", "layer": f"qlinear {n}x{k} -> {m} (int32 out)", "us_kernel": round(t * 1e6, 3),
                      "macs": n * k * m, "algorithmic_bytes": nbytes,
                      "roofline": {"bound": "hbm", "achieved": round(gbs, 1), "peak": pk["hbm_gbs"], "unit": "GB/s",
                                   "frac": round(gbs / pk["hbm_gbs"], 4)},
                      "l2": f"rotating {nsets} buffer sets"}), flush=True)


def run_cifar_pipeline(layers, layer_tensors, graph_time, stream, dev):
    """Config 3 end to end on the device: conv, pool, conv, pool, conv, pool, FC per step."""
    import torch
    from paper_1908_11263_gb300 import qnn
    n = layers[0][1].n
    xin = torch.from_numpy(inputs.cifar_input(n).astype(np.uint8)).to(dev)
    tensors = [layer_tensors(key, layer, wl, lid, with_x=False)[1] for key, layer, wl, lid in layers]
    fw, fb = inputs.cifar_fc()
    fw, fb = torch.from_numpy(fw).to(dev), torch.from_numpy(fb).to(dev)
    bufs = []
    for (_, layer, _, _) in layers:
        bufs.append(torch.empty((n, layer.oh, layer.ow, layer.m), dtype=torch.uint8, device=dev))
        bufs.append(torch.empty((n, layer.oh // 2, layer.ow // 2, layer.m), dtype=torch.uint8, device=dev))
    out = torch.empty((n, 10), dtype=torch.int32, device=dev)

    out_fused = torch.empty_like(out)

    def net(_):
        a = xin
        for li, (_, layer, _, _) in enumerate(layers):
            t = tensors[li]
            qnn.conv_hwc(a, t["w"], t["kappa"], t["lam"], bias=t["bias"], shift=t["shift"], pad=layer.pad,
                         out=bufs[2 * li], stream=stream)
            qnn.maxpool(bufs[2 * li], 2, 2, 8, out=bufs[2 * li + 1], stream=stream)
            a = bufs[2 * li + 1]
        qnn.linear(a.view(n, -1), fw, fb, out=out, stream=stream)

    def net_fused(_):
        # each conv + pool pair as one qconv_hwc_pool2 launch pair (prep + fused kernel)
        a = xin
        for li, (_, layer, _, _) in enumerate(layers):
            t = tensors[li]
            qnn.conv_hwc_pool2(a, t["w"], t["kappa"], t["lam"], bias=t["bias"], shift=t["shift"], pad=layer.pad,
                               out=bufs[2 * li + 1], stream=stream)
            a = bufs[2 * li + 1]
        qnn.linear(a.view(n, -1), fw, fb, out=out_fused, stream=stream)

    # the filters of an inference network prepared once, at set-up (qconv_hwc_prepare); each step is
    # then one qconv_hwc_pool2_run launch per layer and the FC layer
    preps = [qnn.PreparedConv(t["w"], t["kappa"], t["lam"], n=n, h=layer.h, wd=layer.w, bias=t["bias"],
                              shift=t["shift"], bits=8, stride=1, pad=layer.pad, stream=stream)
             for t, (_, layer, _, _) in zip(tensors, layers)]
    out_prepared = torch.empty_like(out)

    def net_prepared(_):
        a = xin
        for li, prep in enumerate(preps):
            prep.pool2(a, out=bufs[2 * li + 1], stream=stream)
            a = bufs[2 * li + 1]
        qnn.linear(a.view(n, -1), fw, fb, out=out_prepared, stream=stream)

    macs = sum(layer.macs for (_, layer, _, _) in layers) + n * 1024 * 10
    with torch.cuda.stream(stream):
        net(0)
        net_fused(0)
        net_prepared(0)
    torch.cuda.synchronize(dev)
    same = bool(torch.equal(out, out_fused)) and bool(torch.equal(out, out_prepared))
    for fn, name in ((net, "cifar_pipeline_n1024 (3 conv + 3 pool + FC, one graph)"),
                     (net_fused, "cifar_pipeline_fused_n1024 (3 fused conv+pool + FC, one graph)"),
                     (net_prepared, "cifar_pipeline_fused_prepared_n1024 (filters prepared once; 3 fused conv+pool "
                                    "runs + FC, one graph)")):
        t_net = graph_time(fn, 20, 5)
        qnn.device_status(stream)
        print(json.dumps({"sweep": "3", "layer": name, "macs": macs, "gmacs_call": round(macs / t_net / 1e9, 1),
                          "us_call": round(t_net * 1e6, 3), "images_per_s": round(n / t_net, 1),
                          "fc_outputs_equal_unfused": same}), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", dest="cpu_baseline", action="store_false")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--sweep", action="store_true", help="per-config measurement lines (workloads 1, 3, 4, 5)")
    ap.add_argument("--no-oracle-times", dest="oracle_times", action="store_false",
                    help="--sweep without the oracle's one-thread and all-core times per layer")
    args = ap.parse_args()
    if args.sweep:
        run_sweep(args)
        return
    if args.impl == "reference":
        # the oracle runs on rank 0's host cores only; other ranks exit without work
        world = int(os.environ.get("WORLD_SIZE", "1"))
        rank = int(os.environ.get("RANK", "0"))
        res = run_reference(args, world, rank)
        if res is not None:
            print(json.dumps(res), flush=True)
        return
    world, rank, local = dist_setup()
    res = run_ours(args, world, rank, local)
    if rank == 0 and res is not None:
        print(json.dumps(res), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
