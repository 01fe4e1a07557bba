#!/usr/bin/env python3
"""Benchmark: the VGG-16 3x3 conv stack, batch 32, fp32, through libpatconv on one GB300 per rank.

One step = the 13 pattern-pruned 3x3 convolutions (bias + ReLU fused; the 2x2 max-pool after
each of the 5 blocks fused into the block's last conv), over one batch of 32 synthetic 3x224x224
images resident in HBM.  Keep ratio
1.0 on the first layer and 0.3 on the others, 8-pattern library, seeded He-normal weights and
N(0,1) images (the paper's trained networks and ImageNet images are not available).

Prints one JSON line (rank 0).  `value` is images/s over all ranks (each rank runs its own
batch: weak scaling, no collective in the data path).  Extra keys:
  roofline      the dominant kernel (pconv_tm) against the FP32 CUDA-core peak
                (SMs x 128 lanes x 2 FLOP x max SM clock), from CUDA events around each of its
                launches inside the timed region;
  e2e           the same metric with every step's input batch copied from pinned host memory
                and its final feature map copied back inside the timed region (the copies on a
                second stream, double-buffered, overlapping the neighbouring steps' compute);
  cpu_baseline  the float64 oracle timed on this host's cores on a bounded sample (rank 0, N=1).
`--impl reference` times the oracle alone as the reference arm.
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "pattern-sparse 3x3 conv useful GFLOP/s & % roofline; VGG-16 img/s at 1 GB300"
BATCH = 32
WORKLOAD = "vgg16_3x3_stack_b32"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=60)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0, help="oracle sample budget")
    ap.add_argument("--profile-layer", type=int, default=None,
                    help="run only layer IDX (0-based) of VGG-16, or of --workload resnet50 / "
                         "mobilenet, --steps times at --batch (for ncu)")
    ap.add_argument("--batch", type=int, default=BATCH, help="batch of --profile-layer")
    ap.add_argument("--workload", choices=["vgg16", "single", "resnet50", "mobilenet"], default="vgg16",
                    help="vgg16: the headline step; the others time each layer of that config alone "
                         "and report it against its roofline")
    ap.add_argument("--sweep", action="store_true", help="single-layer roofline sweep (288 points)")
    ap.add_argument("--sweep-out", default=None, help="also write the sweep as a markdown table here")
    ap.add_argument("--no-dense-context", action="store_true", help="skip the cuDNN dense context")
    return ap.parse_args()


def conv_cost(beta, cin, cout, h, w, ho, wo, n, G, es=4, cin_g=None):
    """Useful FLOP (8 per kept kernel per output pixel) and algorithmic bytes (input and output
    activations once, the packed weight image once, the bias) of one pattern-sparse conv."""
    cin_g = cin if cin_g is None else cin_g
    flops = 8.0 * beta * n * ho * wo
    image = 4 * G * 8 + 8 * G * cin_g + 4 * (G * cin_g + 1) + 16 * beta
    bytes_ = es * (n * cin * h * w + n * cout * ho * wo) + image + 4 * cout
    return flops, float(bytes_)


def config_dict():
    return {"workload": WORKLOAD, "model": "VGG-16 (13 3x3 convs, 5 max-pools)", "batch": BATCH,
            "global_batch": BATCH, "image": "3x224x224", "keep": "1.0 first layer, 0.3 others",
            "patterns": "8 four-tap patterns", "io": "fp32",
            "l2": "no flush: activations per layer up to 411 MB, larger than the 129 MB L2",
            "pool": "2x2 max-pool fused into each block's last conv (pp_conv_pool_ws)",
            "parallelism": "batch replicas"}


# ------------------------------------------------------------------------------ clocks

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *a):
        self.lines = []
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()
                out = ""
            self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        sm, mx, reasons = [], [], set()
        for l in getattr(self, "lines", []):
            parts = [p.strip() for p in l.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for name, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------------------ oracle (CPU)

def blas_threads():
    """Threads of the BLAS numpy runs on (OpenBLAS queried directly), else the usable cores."""
    try:
        with open("/proc/self/maps") as f:
            libs = {l.split()[-1] for l in f if "openblas" in l.lower() and l.split()[-1].startswith("/")}
        for path in libs:
            lib = ctypes.CDLL(path)
            for fn in ("openblas_get_num_threads", "openblas_get_num_threads64_",
                       "scipy_openblas_get_num_threads", "scipy_openblas_get_num_threads64_"):
                if hasattr(lib, fn):
                    return int(getattr(lib, fn)())
    except Exception:
        pass
    return len(os.sched_getaffinity(0))


def set_blas_threads(n):
    """Set OpenBLAS's thread count (numpy's BLAS, found as in blas_threads); False if not found."""
    try:
        with open("/proc/self/maps") as f:
            libs = {l.split()[-1] for l in f if "openblas" in l.lower() and l.split()[-1].startswith("/")}
        for path in libs:
            lib = ctypes.CDLL(path)
            for fn in ("openblas_set_num_threads", "openblas_set_num_threads64_",
                       "scipy_openblas_set_num_threads", "scipy_openblas_set_num_threads64_"):
                if hasattr(lib, fn):
                    getattr(lib, fn)(int(n))
                    return True
    except Exception:
        pass
    return False


def oracle_single_layer(budget_s=10.0):
    """The float64 oracle on the 64->64 32x32 N=1 layer, timed on all BLAS threads and on one:
    [{"threads": t, "ms": median ms}, ...] (projection outside the timed region)."""
    import numpy as np
    from oracle import conv as OC
    from oracle import patterns as OP
    from oracle import project as OPR
    from paper_2003_06513_gb300 import workloads as WL
    L = WL.single_layer()
    Wh = OPR.project(WL.weights(L), OP.default8(), L.keep)["W_hat"]
    b = WL.bias(L).astype(np.float64)
    x = WL.layer_input(L, 1).astype(np.float64)
    full = blas_threads()
    rows = []
    for t in (full, 1):
        if t == 1 and not set_blas_threads(1):
            break
        times, t0 = [], time.perf_counter()
        while len(times) < 30 and (time.perf_counter() - t0 < budget_s or len(times) < 3):
            s0 = time.perf_counter()
            OC.conv_ref(x, Wh, b, 1, True)
            times.append(time.perf_counter() - s0)
        rows.append({"threads": blas_threads(), "ms": 1e3 * statistics.median(times), "runs": len(times)})
    set_blas_threads(full)
    return rows


def oracle_setup(max_images=8):
    """Projected weights of the 13 layers (outside any timed region) and the sample images."""
    from oracle import patterns as OP
    from oracle import project as OPR
    from paper_2003_06513_gb300 import workloads as WL
    layers = WL.vgg16()
    proj = [(OPR.project(WL.weights(L), OP.default8(), L.keep)["W_hat"], WL.bias(L)) for L in layers]
    return layers, proj, WL.vgg16_image(max_images)


def oracle_forward(layers, proj, x):
    """One image batch through the stack: float64 conv over the projected weights + max-pool."""
    import numpy as np
    from oracle import conv as OC
    x = x.astype(np.float64)
    for L, (Wh, b) in zip(layers, proj):
        x = OC.conv_ref(x, Wh, b, 1, True)
        if L.pool_after:
            x = OC.maxpool2x2(x)
    return x


def oracle_forward_images(budget_s, max_images=8):
    """Images pushed through the oracle one at a time until ``budget_s`` elapses;
    returns (images, seconds, threads)."""
    layers, proj, imgs = oracle_setup(max_images)
    t0 = time.perf_counter()
    done = 0
    while done < max_images:
        oracle_forward(layers, proj, imgs[done:done + 1])
        done += 1
        if time.perf_counter() - t0 >= budget_s:
            break
    return done, time.perf_counter() - t0, blas_threads()


def reference_arm(args, rank, world):
    if rank != 0:
        return
    steps, warm = args.steps, args.warmup
    per_step = []
    n_img_total, t_total = 0, 0.0
    threads = blas_threads()
    # each step: one image through the whole stack (bounded sample of the batch-32 workload)
    layers, proj, imgs = oracle_setup(1)
    budget = 240.0
    t_start = time.perf_counter()
    k_done = 0
    for k in range(warm + steps):
        if time.perf_counter() - t_start > budget and k >= warm + 1:
            break
        t0 = time.perf_counter()
        oracle_forward(layers, proj, imgs[:1])
        dt = time.perf_counter() - t0
        if k >= warm:
            per_step.append(dt)
            n_img_total += 1
            t_total += dt
            k_done += 1
    value = n_img_total / t_total if t_total > 0 else 0.0
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "img/s",
            "n_gpus": world, "steps": k_done, "warmup": warm,
            "ms_per_step": 1e3 * t_total / max(k_done, 1), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_dict(),
            "cpu_baseline": {"value": value, "unit": "img/s", "cores": threads, "cpu_count": os.cpu_count(),
                             "kind": "oracle",
                             "sample": "1 image through the 13-layer stack per step (numpy float64)"},
            "e2e": {"value": value, "unit": "img/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------------------ our arm

def fp32_peak(props, clocks):
    """Nominal FP32 CUDA-core peak (context beside the measured one): SMs x 128 FMA lanes x 2 FLOP
    x max SM clock."""
    mhz = None
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            mhz = float(json.load(f).get("sm_max_mhz"))
    except Exception:
        pass
    if not mhz:
        mhz = clocks.get("sm_max_mhz") or 2070.0
    return props.multi_processor_count * 128 * 2 * mhz * 1e6, mhz


_MEASURED_PEAK = {}


def measured_fp32_peak(dev):
    """The FP32 FMA peak measured on this GPU by the library (independent FFMA chains on every SM,
    best of 50 launches of about 2 ms, CUDA events), the clocks sampled meanwhile, and a one-line
    basis; cached per device."""
    import torch
    from paper_2003_06513_gb300 import api
    key = int(getattr(dev, "index", dev) or 0)
    if key not in _MEASURED_PEAK:
        with torch.cuda.device(key), ClockSampler(key) as clk:
            peak = api.measure_fp32_peak(50)
        props = torch.cuda.get_device_properties(key)
        nominal, mhz = fp32_peak(props, {})
        cl = clk.summary()
        basis = (f"measured: FFMA chains on {props.multi_processor_count} SMs, best of 50 x ~2 ms "
                 f"(SM clock median {cl.get('sm_mhz')} MHz); nominal {nominal / 1e12:.1f} TFLOP/s = "
                 f"{props.multi_processor_count} SMs x 128 x 2 x {mhz:.0f} MHz")
        _MEASURED_PEAK[key] = (peak, basis, cl, nominal)
    return _MEASURED_PEAK[key]


def hbm_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]) * 1e9, "measured"
    except Exception:
        return 6.8e12, "fallback"


def kernel_sources_sha256():
    """Hash of the kernel's sources: conv.cu and the channel loop its generator emits."""
    import importlib.util
    csrc = os.path.join(ROOT, "paper_2003_06513_gb300", "csrc")
    spec = importlib.util.spec_from_file_location("gen_dispatch", os.path.join(csrc, "gen_dispatch.py"))
    gen = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(gen)
    h = hashlib.sha256()
    with open(os.path.join(csrc, "conv.cu"), "rb") as f:
        h.update(f.read())
    h.update(gen.generate().encode())
    return h.hexdigest()


def traffic_record():
    """Per-launch DRAM bytes of pconv_tm on this workload from the committed ncu summary, or
    None when the kernel source changed since the counters were taken."""
    path = os.path.join(ROOT, "profiles", "pconv_tm_vgg16_b32_traffic.txt")
    try:
        rec = {}
        with open(path) as f:
            for line in f:
                if ":" in line and not line.startswith("#"):
                    k, v = line.split(":", 1)
                    rec[k.strip()] = v.strip()
        if rec.get("kernel_sources_sha256") == kernel_sources_sha256():
            return {"dram_bytes_per_launch": float(rec["dram_bytes_per_launch"])}
    except Exception:
        pass
    return None


def max_over_ranks(dist, values, device):
    """Each of ``values`` (times measured on this rank) replaced by its maximum over the ranks of
    the process group (the slowest rank sets the job's time); unchanged without a group."""
    import torch
    if dist is None:
        return [float(v) for v in values]
    t = torch.tensor([float(v) for v in values], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.tolist()]


def job_images_per_s(world, ms_per_step):
    """Whole-job throughput: every rank pushes its own batch of BATCH images per step (weak
    scaling), and the step takes the slowest rank's time."""
    return world * BATCH / (ms_per_step * 1e-3)


def our_arm(args, rank, world, local_rank):
    import numpy as np
    import torch
    from paper_2003_06513_gb300 import api
    from paper_2003_06513_gb300 import workloads as WL

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)

    layers = WL.vgg16()
    packed, biases, costs = [], [], []
    shapes = []
    h = 224
    for L in layers:
        lay = api.pp_pack(WL.weights(L), None, L.keep).bind(dev)
        packed.append(lay)
        biases.append(torch.from_numpy(WL.bias(L)).to(dev))
        G = (L.cout + 7) // 8
        fl, by = conv_cost(lay.beta, L.cin, L.cout, h, h, h, h, BATCH, G)
        if L.pool_after:   # the pooled map is what reaches memory
            by -= 4 * BATCH * L.cout * h * h * 3 / 4
        costs.append((fl, by))
        ho = h // 2 if L.pool_after else h
        shapes.append((BATCH, L.cout, ho, ho))
        h = ho
    x0 = torch.from_numpy(WL.vgg16_image(BATCH)).to(dev)
    in_shapes = [(BATCH, L.cin) + ((224, 224) if i == 0 else shapes[i - 1][2:]) for i, L in enumerate(layers)]
    workspace = api.workspace_for(packed, in_shapes, dev, [L.pool_after for L in layers])   # split of small layers
    big = max(int(np.prod(s)) for s in shapes)
    bufA = torch.empty(big, dtype=torch.float32, device=dev)
    bufB = torch.empty(big, dtype=torch.float32, device=dev)
    out_final = torch.empty((BATCH, 512, 7, 7), dtype=torch.float32, device=dev)

    def step(x, ev=None):
        stream = torch.cuda.current_stream(dev)    # the capture stream while a graph records
        cur = x
        bufs = (bufA, bufB)
        j = 0
        for i, (L, lay, b) in enumerate(zip(layers, packed, biases)):
            if i == len(layers) - 1:
                y = out_final
            else:
                y = bufs[j].narrow(0, 0, int(np.prod(shapes[i]))).view(shapes[i])
                j ^= 1
            if ev is not None:
                ev[i][0].record(stream)
            # bias + ReLU fused; a block's last conv also pools 2x2 in its epilogue
            lay.conv(cur, b, True, y, stream, workspace, pool2x2=L.pool_after)
            if ev is not None:
                ev[i][1].record(stream)
            cur = y
        return cur

    def barrier():
        torch.cuda.synchronize(dev)
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize(dev)

    for _ in range(max(args.warmup, 3)):
        step(x0)
    barrier()
    peak_meas, peak_basis, peak_clocks, peak_nominal = measured_fp32_peak(dev)   # the roofline denominator
    barrier()

    K = args.steps
    launches_per_step = len(layers) + sum(
        1 for lay, sh in zip(packed, in_shapes)
        if lay.plan(sh, 0 if workspace is None else workspace.numel() * 4)["splits"] > 1)
    evs = [[[torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)]
            for _ in layers] for _ in range(K)]
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    stream = torch.cuda.current_stream(dev)
    with ClockSampler(dev.index) as clk:
        barrier()
        t0.record(stream)
        for k in range(K):
            step(x0, evs[k])
        t1.record(stream)
        barrier()
    elapsed_ms = t0.elapsed_time(t1)
    conv_ms = [[evs[k][i][0].elapsed_time(evs[k][i][1]) for i in range(len(layers))] for k in range(K)]

    # the same step captured once in a CUDA graph and replayed (no per-launch host work)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step(x0)
    for _ in range(3):
        graph.replay()
    barrier()
    g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    g0.record(stream)
    for _ in range(K):
        graph.replay()
    g1.record(stream)
    barrier()
    graph_ms = g0.elapsed_time(g1) / K

    dense = None
    if not args.no_dense_context:
        dense = dense_context(packed, biases, layers, x0, K, barrier)
    b1_ms, b1_eager = batch1_context(packed, biases, layers, K, barrier, dev)

    # e2e: every step's input batch from pinned host memory and its final feature map back,
    # inside the timed region.  The copies run on a second stream, double-buffered, so that the
    # input of step k+1 and the output of step k-1 move while step k computes; the first input
    # and the last output are not overlapped.
    host_in = torch.from_numpy(WL.vgg16_image(BATCH)).pin_memory()
    host_out = [torch.empty((BATCH, 512, 7, 7), dtype=torch.float32).pin_memory() for _ in range(2)]
    x_dev = [torch.empty_like(x0) for _ in range(2)]
    y_dev = [torch.empty((BATCH, 512, 7, 7), dtype=torch.float32, device=dev) for _ in range(2)]
    copy_stream = torch.cuda.Stream(dev)

    def e2e_run(n_steps):
        ev = lambda: torch.cuda.Event()
        h2d = [ev(), ev()]
        done = [ev() for _ in range(n_steps)]
        d2h = [ev() for _ in range(n_steps)]
        copy_stream.wait_stream(stream)
        with torch.cuda.stream(copy_stream):
            x_dev[0].copy_(host_in, non_blocking=True)
            h2d[0].record(copy_stream)
        for k in range(n_steps):
            b = k & 1
            if k + 1 < n_steps:          # next input, once step k-1 has released that buffer
                with torch.cuda.stream(copy_stream):
                    if k >= 1:
                        copy_stream.wait_event(done[k - 1])
                    x_dev[b ^ 1].copy_(host_in, non_blocking=True)
                    h2d[b ^ 1].record(copy_stream)
            stream.wait_event(h2d[b])
            if k >= 2:                   # the output buffer of step k-2 has been read back
                stream.wait_event(d2h[k - 2])
            y = step(x_dev[b])
            y_dev[b].copy_(y, non_blocking=True)
            done[k].record(stream)
            with torch.cuda.stream(copy_stream):
                copy_stream.wait_event(done[k])
                host_out[b].copy_(y_dev[b], non_blocking=True)
                d2h[k].record(copy_stream)
        stream.wait_event(d2h[n_steps - 1])

    e2e_run(2)
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    Ke = max(2, K // 2)
    e0.record(stream)
    e2e_run(Ke)
    e1.record(stream)
    barrier()
    e2e_ms = e0.elapsed_time(e1) / Ke

    elapsed_ms, e2e_ms, graph_ms = max_over_ranks(dist, [elapsed_ms, e2e_ms, graph_ms], dev)

    if rank == 0:
        clocks = clk.summary()
        peak = peak_meas
        hbm, hbm_kind = hbm_peak()
        flops = [c[0] for c in costs]
        bytes_ = [c[1] for c in costs]
        per_layer_ms = [statistics.median(conv_ms[k][i] for k in range(K)) for i in range(len(layers))]
        tot_conv_ms = sum(statistics.mean(conv_ms[k][i] for k in range(K)) for i in range(len(layers)))
        achieved = sum(flops) / (tot_conv_ms * 1e-3)
        roof_ms = sum(max(f / peak, b / hbm) for f, b in zip(flops, bytes_)) * 1e3
        eager_ms = elapsed_ms / K
        ms_step = min(eager_ms, graph_ms)      # the faster of stream launches and graph replay
        img_s = job_images_per_s(world, ms_step)
        trec = traffic_record()
        line = {
            "metric": METRIC, "value": img_s, "unit": "img/s", "n_gpus": world, "steps": K,
            "warmup": max(args.warmup, 3), "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic (seeded He-normal weights, N(0,1) images)",
            "config": config_dict(),
            "useful_gflops": world * sum(flops) / (ms_step * 1e-3) / 1e9,
            "network_roofline_frac": roof_ms / tot_conv_ms,
            "roofline": {"bound": "alu", "kernel": "pconv_tm<1,float,SORT> (+ split reduce)",
                         "achieved": achieved / 1e12, "peak": peak / 1e12, "unit": "TFLOP/s",
                         "frac": achieved / peak, "peak_kind": "measured", "peak_basis": peak_basis,
                         "peak_nominal": peak_nominal / 1e12, "peak_clocks": peak_clocks,
                         "traffic": (trec or {}).get("dram_bytes_per_launch"),
                         "algorithmic_bytes_per_launch": sum(bytes_) / len(bytes_),
                         "hbm_peak_gbs": hbm / 1e9, "hbm_peak_kind": hbm_kind},
            "timing": {"eager_ms_per_step": eager_ms, "graph_ms_per_step": graph_ms,
                       "value_from": "graph" if graph_ms <= eager_ms else "eager"},
            "per_layer_ms": [round(v, 4) for v in per_layer_ms],
            "e2e": {"value": world * BATCH / (e2e_ms * 1e-3), "unit": "img/s",
                    "h2d_bytes_per_step": int(host_in.numel() * 4),
                    "d2h_bytes_per_step": int(host_out[0].numel() * 4)},
            "gpu_launches": K * launches_per_step,
            "clocks": clocks,
        }
        line["paper_context"] = {
            "note": "the paper's own numbers, for context only: relative speedups of its generated "
                    "mobile code on ResNet-18 (6x compressed), no datacentre-GPU or absolute numbers (§5.3)",
            "device": "Samsung Galaxy S10 (Snapdragon 855: Kryo 485 CPU, Adreno 640 GPU)",
            "speedup_mobile_cpu": {"vs_tflite": 4.2, "vs_tvm": 2.3, "vs_mnn": 2.0},
            "speedup_mobile_gpu": {"vs_tflite": 3.3, "vs_tvm": 2.5, "vs_mnn": 1.4}}
        line["batch1"] = {"value": world * 1.0 / (b1_ms * 1e-3), "unit": "img/s", "ms_per_step": b1_ms,
                          "eager_ms_per_step": b1_eager,
                          "what": "the same 13 layers at batch 1 (latency; graph replay where faster)"}
        if dense is not None:
            line["cudnn_dense_context"] = {"value": world * BATCH / (dense * 1e-3), "unit": "img/s",
                                           "ms_per_step": dense,
                                           "what": "torch conv2d (cuDNN) on the zero-filled projected "
                                                   "weights + bias + ReLU, max_pool2d; fp32, TF32 off"}
        if world == 1 and not args.no_cpu_baseline:
            n, dt, thr = oracle_forward_images(args.cpu_seconds, max_images=BATCH)
            line["cpu_baseline"] = {"value": n / dt, "unit": "img/s", "cores": thr, "cpu_count": os.cpu_count(),
                                    "kind": "oracle",
                                    "sample": f"{n} image(s) through the 13-layer stack, numpy float64"}
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()


def batch1_context(packed, biases, layers, K, barrier, dev):
    """ms per step of the same 13 layers at batch 1 (latency): the smaller of stream launches and
    CUDA-graph replay, with the batch-1 plan's own workspace."""
    import numpy as np
    import torch
    from paper_2003_06513_gb300 import api
    from paper_2003_06513_gb300 import workloads as WL
    x = torch.from_numpy(WL.vgg16_image(1)).to(dev)
    shapes, in_shapes, h = [], [], 224
    for L in layers:
        in_shapes.append((1, L.cin, h, h))
        h = h // 2 if L.pool_after else h
        shapes.append((1, L.cout, h, h))
    ws = api.workspace_for(packed, in_shapes, dev, [L.pool_after for L in layers])
    outs = [torch.empty(sh, dtype=torch.float32, device=dev) for sh in shapes]

    def step():
        cur = x
        for L, lay, b, y in zip(layers, packed, biases, outs):
            lay.conv(cur, b, True, y, torch.cuda.current_stream(dev), ws, pool2x2=L.pool_after)
            cur = y

    for _ in range(3):
        step()
    barrier()
    st = torch.cuda.current_stream(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    Kb = max(10, K)
    e0.record(st)
    for _ in range(Kb):
        step()
    e1.record(st)
    barrier()
    eager = e0.elapsed_time(e1) / Kb
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step()
    for _ in range(3):
        graph.replay()
    barrier()
    e0.record(st)
    for _ in range(Kb):
        graph.replay()
    e1.record(st)
    barrier()
    return min(eager, e0.elapsed_time(e1) / Kb), eager


def dense_context(packed, biases, layers, x0, K, barrier):
    """ms per step of the same network as dense fp32 convolutions (cuDNN) on the zero-filled
    projected weights: the dense work the pattern-sparse path avoids, for context."""
    import torch
    import torch.nn.functional as F
    torch.backends.cudnn.allow_tf32 = False
    torch.backends.cuda.matmul.allow_tf32 = False
    torch.backends.cudnn.benchmark = True
    dev = x0.device
    dense = [torch.from_numpy(lay.export("dense").reshape(L.cout, L.cin_g, 3, 3)).to(dev)
             for lay, L in zip(packed, layers)]

    def dstep(x):
        for L, Wd, b in zip(layers, dense, biases):
            x = F.relu(F.conv2d(x, Wd, b, stride=L.stride, padding=1))
            if L.pool_after:
                x = F.max_pool2d(x, 2)
        return x

    with torch.no_grad():
        for _ in range(3):
            dstep(x0)
        barrier()
        st = torch.cuda.current_stream(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        Kd = max(3, min(K, 20))
        e0.record(st)
        for _ in range(Kd):
            dstep(x0)
        e1.record(st)
        barrier()
    return e0.elapsed_time(e1) / Kd


def _peaks(dev):
    peak, basis, _, _ = measured_fp32_peak(dev)
    hbm, kind = hbm_peak()
    return peak, hbm, kind, basis


def _time_layer(lay, x, b, relu, ws, K, warmup=3):
    """ms of one layer.  Device time: the call captured back to back in one CUDA graph (no host
    work between the launches), cycling through enough copies of x and y that the copies touched
    between two uses of one copy hold more than twice the L2 (each call then reads its input from
    HBM, as the full-size layers do), the graph replayed `warmup` times and then timed with CUDA
    events, divided by the calls.  Also the median of K single stream launches with events around
    each, which includes the host's launch cost where the layer is shorter than that.  Returns
    (ms, eager_ms, graph_ms) with ms = graph_ms."""
    import torch
    y = lay.conv(x, b, relu, workspace=ws)
    for _ in range(warmup - 1):
        lay.conv(x, b, relu, y, workspace=ws)
    torch.cuda.synchronize()
    st = torch.cuda.current_stream()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    for e0, e1 in evs:
        e0.record(st)
        lay.conv(x, b, relu, y, workspace=ws)
        e1.record(st)
    torch.cuda.synchronize()
    eager = statistics.median(e0.elapsed_time(e1) for e0, e1 in evs)
    foot = x.numel() * x.element_size() + y.numel() * y.element_size()
    l2 = getattr(torch.cuda.get_device_properties(x.device), "L2_cache_size", 129 << 20)
    copies = max(1, min(16, -(-2 * l2 // foot)))
    xs = [x] + [x.clone() for _ in range(copies - 1)]
    ys = [y] + [torch.empty_like(y) for _ in range(copies - 1)]
    calls = copies * max(1, -(-8 // copies))
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        for i in range(calls):
            lay.conv(xs[i % copies], b, relu, ys[i % copies], workspace=ws)
    for _ in range(warmup):
        graph.replay()
    torch.cuda.synchronize()
    reps = max(3, K // calls)
    g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    g0.record(st)
    for _ in range(reps):
        graph.replay()
    g1.record(st)
    torch.cuda.synchronize()
    graphed = g0.elapsed_time(g1) / (reps * calls)
    del graph, xs, ys
    return graphed, eager, graphed


def layer_suite(args):
    """Every layer of one config timed alone (inputs resident, larger than L2 where the config is)
    and set against its own roofline min(FP32 peak, AI x HBM bandwidth)."""
    import numpy as np
    import torch
    from paper_2003_06513_gb300 import api
    from paper_2003_06513_gb300 import workloads as WL
    which = args.workload
    if which == "single":
        layers, batch, dt = [WL.single_layer()], 1, "f32"
    elif which == "resnet50":
        layers, batch, dt = WL.resnet50_3x3(), 64, "f32"
    else:
        layers, batch, dt = WL.mobilenet_v2_dw(), 128, "f16"
    tdt, ndt, es = (torch.float16, np.float16, 2) if dt == "f16" else (torch.float32, np.float32, 4)
    peak, hbm, hbm_kind, basis = _peaks(0)
    K = max(args.steps, 30)
    rows, tot_ms, tot_roof, tot_flops = [], 0.0, 0.0, 0.0
    with ClockSampler(0) as clk:
        for L in layers:
            lay = api.pp_pack(WL.weights(L), None, L.keep, groups=L.cout if L.depthwise else 1,
                              stride=L.stride).bind("cuda")
            x = torch.from_numpy(WL.layer_input(L, batch, dtype=ndt)).cuda()
            b = torch.from_numpy(WL.bias(L)).cuda()
            nb = lay.workspace_bytes(x.shape, dtype=x.dtype)
            ws = torch.empty(max(nb // 4, 1), device="cuda") if nb else None
            ms, ms_eager, ms_graph = _time_layer(lay, x, b, True, ws, K, warmup=10)
            G = (L.cout + 7) // 8
            fl, by = conv_cost(lay.beta, L.cin, L.cout, L.h, L.w, L.ho, L.wo, batch, G, es, L.cin_g)
            roof = max(fl / peak, by / hbm) * 1e3
            rows.append({"layer": L.name, "shape": [batch, L.cin, L.h, L.w, L.cout, L.stride], "ms": round(ms, 5),
                         "eager_ms": round(ms_eager, 5), "graph_ms": round(ms_graph, 5),
                         "useful_tflops": fl / ms / 1e9, "gbs": by / ms / 1e6,
                         "bound": "alu" if fl / peak >= by / hbm else "hbm", "roofline_frac": roof / ms,
                         "plan_path": lay.plan(x.shape, nb)["path"]})
            tot_ms += ms
            tot_roof += roof
            tot_flops += fl
            del x, ws
    line = {"metric": METRIC, "workload": which, "value": tot_flops / (tot_ms * 1e-3) / 1e9, "unit": "GFLOP/s",
            "higher_is_better": True, "n_gpus": 1, "steps": K, "dtype": dt, "batch": batch,
            "data": "synthetic (seeded He-normal weights, N(0,1) or post-ReLU inputs)",
            "sum_layer_ms": tot_ms,
            "roofline": {"frac": tot_roof / tot_ms, "fp32_peak_tflops": peak / 1e12, "peak_basis": basis,
                         "hbm_gbs": hbm / 1e9, "hbm_kind": hbm_kind,
                         "note": "time-weighted: sum of per-layer roofline times / sum of measured times"},
            "per_layer": rows, "clocks": clk.summary()}
    if which == "single" and not args.no_cpu_baseline:
        orc = oracle_single_layer()
        line["cpu_baseline"] = {"value": tot_flops / (orc[0]["ms"] * 1e-3) / 1e9, "unit": "GFLOP/s",
                                "cores": orc[0]["threads"], "cpu_count": os.cpu_count(), "kind": "oracle",
                                "sample": "the whole layer, median of up to 30 runs (numpy float64)",
                                "rows": orc}
    print(json.dumps(line), flush=True)


def sweep_run(args):
    """Single-layer sweep: useful GFLOP/s against arithmetic intensity for every point."""
    import torch
    from paper_2003_06513_gb300 import api
    from paper_2003_06513_gb300 import workloads as WL
    peak, hbm, hbm_kind, basis = _peaks(0)
    K = max(3, min(args.steps, 10))
    out = []
    with ClockSampler(0) as clk:
        for L, n, dt in WL.sweep():
            tdt, es = (torch.float16, 2) if dt == "f16" else (torch.float32, 4)
            lay = api.pp_pack(WL.weights(L), None, L.keep).bind("cuda")
            g = torch.Generator(device="cuda")
            g.manual_seed(L.x_seed)
            x = torch.randn((n, L.cin, L.h, L.w), generator=g, device="cuda").to(tdt)
            b = torch.from_numpy(WL.bias(L)).cuda()
            nb = lay.workspace_bytes(x.shape, dtype=x.dtype)
            ws = torch.empty(max(nb // 4, 1), device="cuda") if nb else None
            ms = _time_layer(lay, x, b, True, ws, K)[0]
            fl, by = conv_cost(lay.beta, L.cin, L.cout, L.h, L.w, L.ho, L.wo, n, (L.cout + 7) // 8, es)
            roof = max(fl / peak, by / hbm) * 1e3
            rec = {"c": L.cin, "hw": L.h, "n": n, "keep": L.keep, "io": dt, "ms": ms, "ai": fl / by,
                   "useful_gflops": fl / ms / 1e6, "bound": "alu" if fl / peak >= by / hbm else "hbm",
                   "roofline_frac": roof / ms}
            out.append(rec)
            print(json.dumps(rec), flush=True)
            del x, ws
    clocks = clk.summary()
    if args.sweep_out:
        with open(args.sweep_out, "w") as f:
            f.write("# Single-layer roofline sweep: pattern-sparse 3x3 conv, stride 1, 8 patterns\n\n")
            f.write("Command: `python bench.py --sweep --steps %d --sweep-out %s`\n\n" % (args.steps, args.sweep_out))
            f.write(f"Peaks: FP32 {peak / 1e12:.1f} TFLOP/s ({basis}); HBM {hbm / 1e9:.0f} GB/s ({hbm_kind}). "
                    f"Clocks: {json.dumps(clocks)}\n\n")
            f.write("Inputs N(0,1) generated on the device from the point's seed; weights seeded He-normal. "
                    "ms = device time per call: calls captured back to back in one CUDA graph, cycling "
                    "through copies of x and y that together exceed twice the L2. AI = useful FLOP / "
                    "algorithmic bytes.\n\n")
            f.write("| C | HxW | N | keep | io | ms | AI (FLOP/B) | useful GFLOP/s | bound | roofline frac |\n")
            f.write("|---:|---:|---:|---:|:--|---:|---:|---:|:--|---:|\n")
            for r in out:
                f.write(f"| {r['c']} | {r['hw']} | {r['n']} | {r['keep']} | {r['io']} | {r['ms']:.4f} | "
                        f"{r['ai']:.1f} | {r['useful_gflops']:.0f} | {r['bound']} | {r['roofline_frac']:.3f} |\n")


def profile_layer(args):
    """One layer alone at a chosen batch, for profiler captures on small cases: VGG-16 layer
    IDX, or with --workload resnet50 / mobilenet that suite's layer IDX (MobileNet in fp16)."""
    import numpy as np
    import torch
    from paper_2003_06513_gb300 import api
    from paper_2003_06513_gb300 import workloads as WL
    layers = {"resnet50": WL.resnet50_3x3, "mobilenet": WL.mobilenet_v2_dw}.get(args.workload, WL.vgg16)()
    L = layers[args.profile_layer]
    lay = api.pp_pack(WL.weights(L), None, L.keep, groups=L.cout if L.depthwise else 1,
                      stride=L.stride).bind("cuda")
    ndt = np.float16 if args.workload == "mobilenet" else np.float32
    x = torch.from_numpy(WL.layer_input(L, args.batch, relu=not L.depthwise, dtype=ndt)).cuda()
    b = torch.from_numpy(WL.bias(L)).cuda()
    ws_n = lay.workspace_bytes(x.shape, dtype=x.dtype)
    ws = torch.empty(max(ws_n // 4, 1), device="cuda") if ws_n else None
    y = lay.conv(x, b, True, workspace=ws)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.steps):
        lay.conv(x, b, True, y, workspace=ws)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / max(args.steps, 1)
    flops = 8.0 * lay.beta * args.batch * L.ho * L.wo
    print(json.dumps({"layer": L.name, "batch": args.batch, "ms": ms, "useful_tflops": flops / ms / 1e9,
                      "plan": lay.plan(x.shape, ws_n, dtype=x.dtype)}))


def main():
    args = parse()
    if args.profile_layer is not None:
        profile_layer(args)
        return
    if args.sweep:
        sweep_run(args)
        return
    if args.workload != "vgg16" and args.impl == "ours":
        layer_suite(args)
        return
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        reference_arm(args, rank, world)
        return
    our_arm(args, rank, world, local_rank)


if __name__ == "__main__":
    main()
