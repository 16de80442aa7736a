"""Benchmark: images/s of the fixed-point network evaluation on GB300.

Workload (default): VGG-16 architecture, batch 64 synthetic 224x224x3 N(0,1) images, He-init
weights, first and last layers 16-bit (two-limb path), the rest mixed 4-8 bits; 32 candidate
wordlength plans (seeds 7..38) as in an iterative precision-reduction search.  One step evaluates
one candidate plan on one batch:
  1. FL search + quantization of every weight and bias tensor at the plan's wordlengths,
  2. calibration of every activation FL on the 8-image calibration slice (forward-optimizer order),
  3. the integer-only forward of the whole batch through fxpq_net_forward.
value = batch / step time (images per second), whole job over N GPUs (weak scaling: each rank
evaluates its own plans on its own batch; no collective on the data path).

Prints one JSON line (rank 0).  --impl reference times the CPU oracle on a bounded sample.
"""
from __future__ import annotations

import argparse
import ctypes
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

WORKLOADS = {
    "vgg16": {"arch": "vgg16", "batch": 64, "seed": 7, "plans": list(range(7, 39)), "calib": 8},
    "alexnet": {"arch": "alexnet", "batch": 256, "seed": 5, "plans": [5], "calib": 8},
    "resnet18": {"arch": "resnet18", "batch": 128, "seed": 6, "plans": [6], "calib": 8},
    # ResNet-18 with its BN layers kept as Scale layers (bias-free convs), the paper's form
    "resnet18_bn": {"arch": "resnet18_bn", "batch": 128, "seed": 6, "plans": [6], "calib": 8},
}


def device_params(arch, seed, dev):
    """Seeded fp32 parameters on the device: conv name -> (weight, bias or None), BN conv name ->
    (gamma, beta, mean, var)."""
    import torch
    W = synth.weights(arch, seed)
    wdev = {nm: (torch.from_numpy(w).to(dev), None if b is None else torch.from_numpy(b).to(dev))
            for nm, (w, b) in W.items()}
    bn = {nm: tuple(torch.from_numpy(t).to(dev) for t in v) for nm, v in synth.bn_params(arch, seed + 100).items()}
    return wdev, bn
L2_BYTES = 129 * 1024 * 1024


def dist_env():
    r = int(os.environ.get("RANK", "0"))
    w = int(os.environ.get("WORLD_SIZE", "1"))
    lr = int(os.environ.get("LOCAL_RANK", "0"))
    return r, w, lr


class ClockSampler:
    """nvidia-smi samples during the timed region (SM clock, max clock, throttle reasons): one
    streaming nvidia-smi process (-lms 25), started ahead of the region; only the samples stamped
    inside the region are kept."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.samples = []  # (monotonic time, fields)
        self._p = None
        self._t = None
        self.t0 = self.t1 = None

    def _run(self):
        for line in self._p.stdout:
            f = [x.strip() for x in line.strip().split(",")]
            if len(f) >= 7:
                self.samples.append((time.monotonic(), f))

    def __enter__(self):
        try:
            self._p = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                                        "--format=csv,noheader,nounits", "-lms", "25"],
                                       stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self._t = threading.Thread(target=self._run, daemon=True)
            self._t.start()
            deadline = time.monotonic() + 3.0
            while not self.samples and time.monotonic() < deadline:
                time.sleep(0.01)
        except Exception:
            self._p = None
        self.t0 = time.monotonic()
        return self

    def __exit__(self, *a):
        self.t1 = time.monotonic()
        time.sleep(0.05)  # let the sample that straddles the end arrive
        if self._p:
            self._p.terminate()
            try:
                self._p.wait(timeout=5)
            except Exception:
                self._p.kill()
        if self._t:
            self._t.join(timeout=5)

    def summary(self):
        inside = [f for t, f in self.samples if self.t0 <= t <= self.t1 + 0.03]
        if not inside:  # a region shorter than the sampling interval: the nearest samples
            inside = [f for t, f in self.samples[-2:]]
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        sm = [float(s[0]) for s in inside if s[0].replace(".", "").isdigit()]
        mx = [float(s[1]) for s in inside if s[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for s in inside for i in range(4) if len(s) > 3 + i and s[3 + i] == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(inside)}


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d.get("hbm_gbs", 6800.0), d.get("bf16_tflops", 1900.0), d.get("bf16_tflops_sustained", 1700.0), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


def max_over_ranks(ms: float, world: int, device) -> float:
    """The slowest rank's mean step time: every rank times the same number of steps after one barrier."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(world: int, batch: int, t_max_ms: float) -> float:
    """Whole-job images/s: every rank evaluates its own batch (replicas, weak scaling) in t_max."""
    return world * batch / (t_max_ms / 1e3)


# ----------------------------------------------------------------------------- GPU arm
def run_fxpq(args):
    import torch
    import torch.distributed as dist

    rank, world, lrank = dist_env()
    if world > 1:
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(lrank)
    dev = torch.device("cuda", lrank)
    import __graft_entry__ as g
    g.build()
    from paper_2203_12091_gb300 import fxpq as F
    from paper_2203_12091_gb300.net import QNet

    wl = WORKLOADS[args.workload]
    arch, B = wl["arch"], wl["batch"]
    layers = synth.ARCHS[arch]()
    imgs_np = synth.images(B, wl["seed"] + 1000 * rank)
    plans = [synth.bit_plan(arch, s) for s in wl["plans"]]
    wdev, bndev = device_params(arch, wl["seed"], dev)
    imgs = torch.from_numpy(imgs_np).to(dev)
    pinned = torch.from_numpy(imgs_np).pin_memory()
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device=dev)

    def step(i, images):
        q = QNet(layers, hw=224, cin=3)
        q._dev = dev
        plan = plans[(i + rank) % len(plans)]
        q.quantize_params(wdev, plan, None, bndev)
        q.calibrate(images[: wl["calib"]], plan)
        logits, s = q.forward(images)
        return q, logits, s

    for i in range(args.warmup):
        step(i, imgs)
    torch.cuda.synchronize()

    # ---- timed region (device-resident inputs): per-step CUDA events, L2 flushed between steps
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    launches0 = F.fxpq_launch_count()
    times = []
    with ClockSampler(lrank) as clk:
        for i in range(args.steps):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            step(args.warmup + i, imgs)
            e1.record(stream)
            e1.synchronize()
            times.append(e0.elapsed_time(e1))
    torch.cuda.synchronize()
    launches = F.fxpq_launch_count() - launches0
    ms = sum(times) / len(times)
    t_max = max_over_ranks(ms, world, dev)
    value = job_throughput(world, B, t_max)

    # ---- end to end through the public API: pinned host images in, logits out, every step
    e2e_times = []
    for i in range(max(2, min(args.steps, 5))):
        flush.zero_()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        dimgs = pinned.to(dev, non_blocking=True)
        q, logits, s = step(args.warmup + i, dimgs)  # the plans of the first timed steps
        host_logits = logits.cpu()
        torch.cuda.synchronize()
        e2e_times.append(time.perf_counter() - t0)
    e2e_s = sum(e2e_times) / len(e2e_times)
    h2d = pinned.numel() * 4
    d2h = host_logits.numel() * 8

    # ---- roofline of the dominant kernel (the conv C-Block): op-by-op forward with events per conv, on
    # the workload's first plan (the network `--kernel forward` builds, whose conv launches the DRAM
    # traffic capture profiles; another plan's formats can change a layer's exact groups)
    q = QNet(layers, hw=224, cin=3)
    q._dev = dev
    q.quantize_params(wdev, plans[0], None, bndev)
    q.calibrate(imgs[: wl["calib"]], plans[0])
    conv_ms, conv_flops, nconv, conv_layers = conv_roofline(q, imgs, F, stream)
    hbm, bf16, bf16s, src = measured_peaks()
    achieved = conv_flops / (conv_ms / 1e3) / 1e12
    traffic = None
    tpath = os.path.join(ROOT, "profiles", "traffic.json")
    if os.path.exists(tpath):
        traffic = json.load(open(tpath)).get(args.workload)

    if rank == 0:
        cpu = cpu_baseline(args.workload) if (world == 1 and not args.no_cpu) else None
        line = {
            "metric": "images/s for fixed-point net forward (one candidate plan evaluated per step)",
            "value": round(value, 2), "unit": "images/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(t_max, 3), "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "int (exact integer codes; fp16-valued operands)", "data": "synthetic",
            "config": workload_config(args.workload, world),
            "e2e": {"value": round(world * B / e2e_s, 2), "unit": "images/s", "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h},
            "gpu_launches": int(launches),
            "roofline": {"bound": "tensor", "kernel": "conv C-Block", "achieved": round(achieved, 3),
                         "peak": bf16, "unit": "TFLOP/s", "frac": round(achieved / bf16, 5), "traffic": traffic,
                         "peak_source": f"{src} bf16 dense burst (fp16 operands run at the bf16 rate)",
                         "conv_launches_timed": nconv, "conv_layers_us": conv_layers},
            "clocks": clk.summary(),
            "cpu_baseline": cpu,
        }
        print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()


def conv_roofline(q, imgs, F, stream, iters=3):
    """Average conv launch time over `iters` op-by-op forwards (CUDA events on the launching stream).

    A device-side sleep of about 1 ms is queued ahead of each timed conv, so that the host's argument
    preparation (workspace queries, tensor-map encoding, the split reduction's workspace) overlaps it
    and the events bracket the conv kernel(s) alone rather than the host gap before the launch.  The
    first forward is not counted (its allocations reach the device).  Returns the total time, the
    algorithmic FLOPs, the number of timed launches and the per-layer average in microseconds."""
    import torch
    tot_ms, flops, n = 0.0, 0, 0
    per_layer = {}
    N = imgs.shape[0]
    env = None
    for it in range(iters):
        # the previous forward's tensors go back to the caching allocator before this one allocates, so
        # from the second forward on no layer's output allocation reaches the device inside its events
        env = None
        fin = q.fmts["input"]["a"]
        x0 = torch.empty(N * q.hw * q.hw * q.cp_in * F.planes(fin), dtype=torch.float16, device=imgs.device)
        F.fxpq_quantize_images(imgs, fin, q.cp_in, x0)
        env = {"input": (x0, fin)}
        last = len(q.layers) - 1
        for i, L_ in enumerate(q.layers):
            nm = L_["name"]
            mode = F.OUT_ACC64 if i == last else F.OUT_CODES
            if L_["type"] == "conv":
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                torch.cuda._sleep(2_000_000)  # ~1 ms at 2 GHz: longer than the host work of run_layer
                e0.record(stream)
                y, s = q.run_layer(i, env, N, mode)
                e1.record(stream)
                e1.synchronize()
                if it > 0:
                    tot_ms += e0.elapsed_time(e1)
                    per_layer[nm] = per_layer.get(nm, 0.0) + e0.elapsed_time(e1) * 1e3 / (iters - 1)
                    H, _, K = q.shapes[nm]
                    flops += 2 * N * H * H * K * L_["C"] * L_["R"] * L_["R"]
                    n += 1
            else:
                y, s = q.run_layer(i, env, N, mode)
            env[nm] = (y, q.fmts[nm].get("a"))
    return tot_ms, flops, n, {k: round(v, 1) for k, v in per_layer.items()}


# ----------------------------------------------------------------------------- configs 1 and 2
CONFIG1 = {"N": 8, "H": 32, "C": 64, "K": 64, "R": 3}  # 3x3 conv, stride 1, pad 1, 8-bit w/a, FL in 0..15


def config1_inputs():
    """The single-conv workload: ReLU(N(0,1)) NHWC inputs, He-normal KRSC weights (std sqrt(2/576)),
    N(0, 0.01) biases, seeded."""
    c = CONFIG1
    x = np.maximum(synth.normal(c["N"] * c["H"] * c["H"] * c["C"], 1), np.float32(0)).reshape(c["N"], c["H"], c["H"], c["C"])
    w = synth.normal(c["K"] * c["R"] * c["R"] * c["C"], 2, std=float(np.sqrt(2.0 / (c["R"] * c["R"] * c["C"])))).reshape(
        c["K"], c["R"], c["R"], c["C"])
    b = synth.normal(c["K"], 3, std=0.01)
    return x, w, b


def oracle_config1():
    """The oracle running the single-conv workload: FL searches of x, w (k = 8, FL 0..15) and b (k = 16,
    FL -8..23), quantization, the C-Block to its fp32 image, the output FL search, the requantized codes."""
    import oracle
    x, w, b = config1_inputs()
    t0 = time.perf_counter()
    fmts = []
    for t, k, lo, hi in ((x, 8, 0, 15), (w, 8, 0, 15), (b, 16, -8, 23)):
        _, best, S, _ = oracle.fl_search(t, -1, k, k, lo, hi)
        fmts.append((k, S, int(best[0])))
    (kx, Sx, flx), (kw, Sw, flw), (kb, Sb, flb) = fmts
    xq, wq, bq = oracle.quantize(x, kx, Sx, flx), oracle.quantize(w, kw, Sw, flw), oracle.quantize(b, kb, Sb, flb)
    acc = oracle.conv2d(xq.reshape(x.shape), wq.reshape(w.shape), 1, 1)
    v, sc = oracle.cblock(acc, flx + flw, bq, flb, True)
    _, best, Sy, _ = oracle.fl_search(oracle.to_f32(v, sc), -1, 8, 8, 0, 15)
    oracle.requant(v, sc, 8, Sy, int(best[0]))
    return time.perf_counter() - t0


def oracle_config2(n, sweep):
    import oracle
    x = synth.sweep_tensor("normal", n, 2)
    t0 = time.perf_counter()
    if sweep:
        oracle.fl_search(x, -1, 2, 16, -8, 23)
    else:
        oracle.fl_search(x, -1, 8, 8, -8, 23)
    return time.perf_counter() - t0


def oracle_job(spec):
    """Time one oracle job (run in a subprocess with OMP_NUM_THREADS set by the caller)."""
    kind, *a = spec.split(":")
    if kind == "config1":
        t = oracle_config1()
    else:
        t = oracle_config2(int(a[0]), a[1] == "sweep")
    print(json.dumps({"oracle_s": t}))


def timed_oracle(spec, threads):
    """Seconds of an oracle job on `threads` host cores (a subprocess, so that OpenMP reads its count)."""
    env = dict(os.environ, OMP_NUM_THREADS=str(threads))
    r = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-job", spec], capture_output=True,
                       text=True, env=env, timeout=900)
    return json.loads(r.stdout.strip().splitlines()[-1])["oracle_s"]


def bench_config1(args, F):
    """The single-conv workload end to end on the GPU (FL searches of x, w and b as one batch, their
    quantization, the C-Block's fp32 image and its FL search, the requantized codes) and the final
    C-Block alone; the oracle on the same workload on one and on all host cores."""
    import torch
    import paper_2203_12091_gb300._lib as L
    c = CONFIG1
    x, w, b = config1_inputs()
    xd, wd, bd = (torch.from_numpy(np.ascontiguousarray(t)).cuda().reshape(-1) for t in (x, w, b))
    dev = xd.device
    N, H, C, K, R = c["N"], c["H"], c["C"], c["K"], c["R"]
    REC = 64
    res = torch.empty(3 * REC, dtype=torch.uint8, device=dev)
    err = torch.empty(3 * 32, dtype=torch.float64, device=dev)
    ws = F.workspace(F.fxpq_fl_search_batch_workspace(3), dev)
    xq = torch.empty(xd.numel(), dtype=torch.float16, device=dev)
    wq = torch.empty(wd.numel(), dtype=torch.float16, device=dev)
    bq = torch.empty(K, dtype=torch.int32, device=dev)
    y32 = torch.empty(N * H * H * K, dtype=torch.float32, device=dev)
    y = torch.empty(N * H * H * K, dtype=torch.float16, device=dev)
    flops = 2 * N * H * H * K * C * R * R

    def search(items):
        batch = [L.FlSearchItem(t.data_ptr(), t.numel(), -1, k, k, lo, hi, err.data_ptr() + 8 * 32 * i,
                                res.data_ptr() + REC * i, res.data_ptr() + REC * i + 8)
                 for i, (t, k, lo, hi) in enumerate(items)]
        F.fxpq_fl_search_batch(batch, ws)
        host = bytes(res.cpu().numpy().tobytes())
        out = []
        for i, (t, k, lo, hi) in enumerate(items):
            best = int.from_bytes(host[REC * i:REC * i + 4], "little", signed=True)
            st = L.Stats.from_buffer_copy(host[REC * i + 8:REC * i + 8 + ctypes.sizeof(L.Stats)])
            out.append(F.fmt(k, st.is_signed, best))
        return out

    state = {}

    def step():
        fx, fw, fb = search([(xd, 8, 0, 15), (wd, 8, 0, 15), (bd, 16, -8, 23)])
        F.fxpq_quantize(xd, fx, F.DT_F16, xq)
        F.fxpq_quantize(wd, fw, F.DT_F16, wq)
        F.fxpq_quantize(bd, fb, F.DT_I32, bq)
        d32 = F.conv_desc(N, H, H, C, C, K, R, R, 1, 1, True, F.OUT_F32, fx, fw, fb, F.fmt(8, 0, 0))
        F.fxpq_conv_fwd(d32, xq, wq, bq, y32)
        (fy,) = search([(y32, 8, 0, 15)])
        d = F.conv_desc(N, H, H, C, C, K, R, R, 1, 1, True, F.OUT_CODES, fx, fw, fb, fy)
        F.fxpq_conv_fwd(d, xq, wq, bq, y)
        state["d"] = d

    def timeit(fn):
        ts = []
        for i in range(args.warmup + args.steps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            fn()
            e1.record()
            e1.synchronize()
            if i >= args.warmup:
                ts.append(e0.elapsed_time(e1))
        return sum(ts) / len(ts)

    ms_step = timeit(step)
    d = state["d"]
    ms_conv = timeit(lambda: F.fxpq_conv_fwd(d, xq, wq, bq, y))
    hbm, bf16, _, src = measured_peaks()
    t1 = timed_oracle("config1", 1)
    tn = timed_oracle("config1", os.cpu_count() or 1)
    return {"config1": {
        "workload": "3x3 conv, batch 8, 64->64 channels, 32x32 maps, 8-bit w/a (FL 0..15), 16-bit bias, 8-bit output",
        "step_ms": round(ms_step, 4), "conv_us": round(ms_conv * 1e3, 2),
        "conv_tops": round(flops / (ms_conv / 1e3) / 1e12, 2), "conv_frac_peak": round(flops / (ms_conv / 1e3) / 1e12 / bf16, 4),
        "peak_tflops": bf16, "peak_source": src,
        "oracle_step_s_1_thread": round(t1, 3), "oracle_step_s_all_cores": round(tn, 3), "host_cores": os.cpu_count()}}


def bench_config2(args, F):
    """The FL-search sweep workload: per size (1M, 16M, 64M) and distribution (N(0,1), Laplace(0, 0.1),
    ReLU(N(0,1))) the single-wordlength search (k = 8, FL -8..23), the full 15 x 32 grid (k 2..16) and the
    quantization to int8 codes; the oracle on 1M (row and grid) and 16M (row) values."""
    import torch
    hbm, _, _, src = measured_peaks()
    rows = []
    for n in (1 << 20, 1 << 24, 1 << 26):
        for dist in ("normal", "laplace", "relu_normal"):
            x = torch.from_numpy(synth.sweep_tensor(dist, n, 2)).cuda()
            y = torch.empty(n, dtype=torch.int8, device="cuda")
            r = {"n": n, "dist": dist}
            for name, fn in (("row_k8", lambda: F.fl_search(x, -1, 8, 8, -8, 23)),
                             ("grid_k2_16", lambda: F.fl_search(x, -1, 2, 16, -8, 23)),
                             ("quantize_i8", lambda: F.fxpq_quantize(x, F.fmt(8, 1, 5), F.DT_I8, y))):
                ts = []
                for i in range(args.warmup + args.steps):
                    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    e0.record()
                    fn()
                    e1.record()
                    e1.synchronize()
                    if i >= args.warmup:
                        ts.append(e0.elapsed_time(e1))
                ms = sum(ts) / len(ts)
                nbytes = (5 if name == "quantize_i8" else 4) * n
                r[name] = {"ms": round(ms, 4), "gelem_s": round(n / (ms / 1e3) / 1e9, 1),
                           "gbs": round(nbytes / (ms / 1e3) / 1e9, 1), "frac_hbm": round(nbytes / (ms / 1e3) / 1e9 / hbm, 3)}
            rows.append(r)
    cores = os.cpu_count() or 1
    orc = {"row_1M_s_1_thread": round(timed_oracle(f"config2:{1 << 20}:row", 1), 3),
           "row_1M_s_all_cores": round(timed_oracle(f"config2:{1 << 20}:row", cores), 3),
           "grid_1M_s_all_cores": round(timed_oracle(f"config2:{1 << 20}:sweep", cores), 3),
           "row_16M_s_all_cores": round(timed_oracle(f"config2:{1 << 24}:row", cores), 3), "host_cores": cores}
    return {"config2": {"rows": rows, "hbm_gbs": hbm, "peak_source": src, "oracle": orc}}


# ----------------------------------------------------------------------------- CPU oracle arm
def oracle_step(workload, n_images=1):
    """The oracle evaluating one candidate plan on a bounded sample: parameter FL search and
    quantization, calibration on a 1-image slice, forward of `n_images` images."""
    import oracle.net as onet
    wl = WORKLOADS[workload]
    arch = wl["arch"]
    layers = synth.ARCHS[arch]()
    W = synth.weights(arch, wl["seed"])
    bn = synth.bn_params(arch, wl["seed"] + 100)
    imgs = synth.images(n_images, wl["seed"])
    plan = synth.bit_plan(arch, wl["plans"][0])
    t0 = time.perf_counter()
    fm, qp = onet.calibrate(layers, W, imgs[:1], plan, bn)
    onet.forward(layers, fm, qp, imgs)
    return time.perf_counter() - t0


def cpu_baseline(workload):
    t = oracle_step(workload, 1)
    cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    return {"value": round(1.0 / t, 5), "unit": "images/s", "cores": cores, "kind": "oracle",
            "sample": f"{workload}: one candidate plan -- parameter FL search + quantize, calibration on a "
                      f"1-image slice, forward of 1 image ({t:.1f} s)"}


def workload_config(workload, world):
    """The bench line's `config` (both arms): the workload and how it is laid out over the ranks."""
    wl = WORKLOADS[workload]
    return {"workload": f"{wl['arch']} batch {wl['batch']}, {len(wl['plans'])} candidate plans, calib slice {wl['calib']}",
            "model": wl["arch"], "global_batch": wl["batch"] * world, "seq_len": None,
            "parallelism": f"replicas x{world}", "l2": "flushed between timed steps (2x L2 buffer written)"}


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    ts = [oracle_step(args.workload, 1) for _ in range(args.warmup)]
    ts = [oracle_step(args.workload, 1) for _ in range(args.steps)]
    t = sum(ts) / len(ts)
    cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    v = round(1.0 / t, 5)
    print(json.dumps({
        "impl": "reference", "metric": "images/s for fixed-point net forward (one candidate plan evaluated per step)",
        "value": v, "unit": "images/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(t * 1e3, 1), "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "int64 (exact)", "data": "synthetic",
        "config": workload_config(args.workload, world),
        "cpu_baseline": {"value": v, "unit": "images/s", "cores": cores, "kind": "oracle",
                         "sample": f"{args.workload}, rank 0 on the host cores: per step one candidate plan -- "
                                   "parameter FL search + quantize, calibration on a 1-image slice, forward of "
                                   "1 image"},
        "e2e": {"value": v, "unit": "images/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


def run_kernel(args):
    """Single-kernel timing cases (also the targets of the ncu captures summarised in profiles/):
    conv     : VGG-16 conv3_1-shaped C-Block, batch 64, 56x56x128 -> 256, 3x3 pad 1, 8-bit codes, with
               and without the weight-code L1 bound;
    flsearch : FL search over 64M N(0,1) fp32 values, one wordlength (k=8) and the full 15 x 32 grid, with
               the L2 score and with the L1 score (k = 1..16 for the sweep);
    quantize : Q of 64M N(0,1) fp32 values to int8 codes and to an fp16 code tensor (HBM-bound);
    fopt     : the forward optimizer (Alg. 1, cost F) on ResNet-18 with 8 calibration images, and its fp32
               convolution;
    forward  : the integer forward of the workload (first plan, calibrated once), fxpq_net_forward alone."""
    import torch
    import __graft_entry__ as g
    g.build()
    from paper_2203_12091_gb300 import fxpq as F
    out = {}
    if args.kernel in ("conv", "all"):
        N, H, C, K = 64, 56, 128, 256
        rng = np.random.default_rng(0)
        x = torch.from_numpy(rng.integers(0, 256, size=(N, H, H, C)).astype(np.float16)).cuda()
        w = torch.from_numpy((rng.integers(-128, 128, size=(K, 3, 3, C)) // 4).astype(np.float16)).cuda()
        b = torch.from_numpy(rng.integers(-2 ** 15, 2 ** 15, size=K).astype(np.int32)).cuda()
        y = torch.empty(N * H * H * K, dtype=torch.float16, device="cuda")
        l1 = torch.zeros(1, dtype=torch.int64, device="cuda")
        F.fxpq_code_l1max(w, K, 9 * C, l1)
        # "conv": groups from the wordlength bound alone; "conv_l1": with the weight-code L1 bound
        for name, w_l1 in (("conv", 0), ("conv_l1", int(l1.item()))):
            d = F.conv_desc(N, H, H, C, C, K, 3, 3, 1, 1, 1, F.OUT_CODES, F.fmt(8, 0, 4), F.fmt(8, 1, 8),
                            F.fmt(16, 1, 18), F.fmt(8, 0, 3), w_l1)
            ts = []
            for i in range(args.warmup + args.steps):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                F.fxpq_conv_fwd(d, x, w, b, y)
                e1.record()
                e1.synchronize()
                if i >= args.warmup:
                    ts.append(e0.elapsed_time(e1))
            ms = sum(ts) / len(ts)
            out[name] = {"ms": round(ms, 4), "tflops": round(2 * N * H * H * K * C * 9 / (ms / 1e3) / 1e12, 2)}
    if args.kernel in ("flsearch", "all"):
        n = 1 << 26
        x = torch.from_numpy(synth.normal(n, 2)).cuda()
        for name, (klo, khi, score) in (("flsearch_k8", (8, 8, "l2")), ("flsearch_sweep", (2, 16, "l2")),
                                        ("flsearch_k8_l1", (8, 8, "l1")), ("flsearch_sweep_l1", (1, 16, "l1"))):
            ts = []
            for i in range(args.warmup + args.steps):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                F.fl_search(x, -1, klo, khi, -8, 23, score=score)
                e1.record()
                e1.synchronize()
                if i >= args.warmup:
                    ts.append(e0.elapsed_time(e1))
            ms = sum(ts) / len(ts)
            out[name] = {"ms": round(ms, 4), "gelem_s": round(n / (ms / 1e3) / 1e9, 2),
                         "hbm_gbs": round(4 * n / (ms / 1e3) / 1e9, 1)}
    if args.kernel in ("quantize", "all"):
        # Q on 64M fp32 values: 4 B read + 1 B (int8 codes) or 2 B (fp16 code tensor) written per value
        n = 1 << 26
        x = torch.from_numpy(synth.normal(n, 2)).cuda()
        hbm = measured_peaks()[0]
        for name, dt, bw in (("quantize_i8", F.DT_I8, 1), ("quantize_f16", F.DT_F16, 2)):
            y = torch.empty(n * bw, dtype=torch.uint8, device="cuda")
            ts = []
            for i in range(args.warmup + args.steps):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                F.fxpq_quantize(x, F.fmt(8, 1, 5), dt, y)
                e1.record()
                e1.synchronize()
                if i >= args.warmup:
                    ts.append(e0.elapsed_time(e1))
            ms = sum(ts) / len(ts)
            gbs = (4 + bw) * n / (ms / 1e3) / 1e9
            out[name] = {"ms": round(ms, 4), "gbs": round(gbs, 1), "frac_hbm": round(gbs / hbm, 3)}
    if args.kernel in ("quantize", "all"):
        # packed k-bit storage of 64M 4-bit codes: 2 B read + 0.5 B written per code (pack), the reverse
        # for unpack
        n = 1 << 26
        f4 = F.fmt(4, 1, 0)
        codes = torch.randint(-8, 8, (n,), dtype=torch.int32, device="cuda").to(torch.float16)
        words = torch.empty(F.packed_words(n, f4), dtype=torch.int32, device="cuda")
        hbm = measured_peaks()[0]
        for name, fn in (("pack_k4", lambda: F.fxpq_pack_codes(codes, n, f4, words)),
                         ("unpack_k4", lambda: F.fxpq_unpack_codes(words, n, f4, codes))):
            ts = []
            for i in range(args.warmup + args.steps):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                fn()
                e1.record()
                e1.synchronize()
                if i >= args.warmup:
                    ts.append(e0.elapsed_time(e1))
            ms = sum(ts) / len(ts)
            gbs = 2.5 * n / (ms / 1e3) / 1e9
            out[name] = {"ms": round(ms, 4), "gbs": round(gbs, 1), "frac_hbm": round(gbs / hbm, 3)}
    if args.kernel in ("fopt", "all"):
        # the forward optimizer (Alg. 1 with the cost F) on ResNet-18, 8 calibration images at 224 x 224:
        # the first 12 data-structures, every candidate's cost over the whole network
        from paper_2203_12091_gb300.fopt import ForwardOptimizer
        wdev, _ = device_params("resnet18", 6, torch.device("cuda"))
        imgs = torch.from_numpy(synth.images(8, 6)).cuda()
        plan = synth.bit_plan("resnet18", 6)
        t0 = time.perf_counter()
        fo = ForwardOptimizer(synth.resnet18(), wdev, imgs, plan)
        torch.cuda.synchronize()
        t_init = time.perf_counter() - t0
        n_eval = [0]
        costs0 = fo.costs

        def counted(cur, fls):
            n_eval[0] += len(fls)
            return costs0(cur, fls)

        fo.costs = counted
        t0 = time.perf_counter()
        res = fo.run(1, 12)
        torch.cuda.synchronize()
        dt = time.perf_counter() - t0
        out["fopt"] = {"workload": "resnet18 224x224, 8 calibration images, K=1, first 12 data-structures",
                       "init_s": round(t_init, 3), "s": round(dt, 3), "cost_evals": n_eval[0],
                       "ms_per_cost_eval": round(1e3 * dt / max(n_eval[0], 1), 2),
                       "note": "candidates of one data-structure share a batched forward",
                       "data_structures_s": round(len(res) / dt, 2)}
        # the fp32 convolution of the FP32 side on a ResNet-18 stage-2 shape: 8 x 56 x 56 x 64 -> 64, 3 x 3
        N, H, C, K = 8, 56, 64, 64
        x = torch.randn(N * H * H * C, device="cuda")
        w = torch.randn(K * 9 * C, device="cuda")
        y = torch.empty(N * H * H * K, device="cuda")
        ts = []
        for i in range(args.warmup + args.steps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            F.fxpq_conv_f32(N, H, H, C, K, 3, 3, 1, 1, True, x, w, None, y)
            e1.record()
            e1.synchronize()
            if i >= args.warmup:
                ts.append(e0.elapsed_time(e1))
        ms = sum(ts) / len(ts)
        tf = 2.0 * N * H * H * K * 9 * C / (ms / 1e3) / 1e12
        peak = 152 * 128 * 2 * 2.07e9 / 1e12  # fp32 FMA lanes x 2 FLOP x max SM clock
        out["conv_f32"] = {"ms": round(ms, 4), "tflops": round(tf, 2), "peak_fp32_tflops": round(peak, 1),
                           "frac": round(tf / peak, 3)}
    if args.kernel in ("fc", "all"):
        # VGG-16 fc6 at batch 64 (25088 -> 4096: a 7 x 7 kernel over the 7 x 7 map) with k-bit weights read
        # as fp16 code tensors and as packed k-bit planes (Sec. V-E.2); weight bytes read per launch
        N, H, C, K = 64, 7, 512, 4096
        rng = np.random.default_rng(5)
        x = torch.from_numpy(rng.integers(0, 32, size=(N, H, H, C)).astype(np.float16)).cuda()
        b = torch.from_numpy(rng.integers(-2 ** 15, 2 ** 15, size=K).astype(np.int32)).cuda()
        y = torch.empty(N * K, dtype=torch.float16, device="cuda")
        for kw in (8, 4):
            wc = rng.integers(-(1 << (kw - 1)), 1 << (kw - 1), size=(K, H, H, C))
            w = torch.from_numpy(wc.astype(np.float16)).cuda()
            fw = F.fmt(kw, 1, kw + 4)
            l1 = int(np.abs(wc).reshape(K, -1).sum(axis=1).max())
            wp = F.pack_weights(w, fw, K, H * H * C)
            for name, packed in ((f"fc6_k{kw}_f16", None), (f"fc6_k{kw}_packed", wp)):
                d = F.conv_desc(N, H, H, C, C, K, H, H, 1, 0, 1, F.OUT_CODES, F.fmt(5, 0, 2), fw, F.fmt(16, 1, 20),
                                F.fmt(8, 0, 3), l1, wpacked=packed)
                ws = torch.empty(F.fxpq_conv_workspace(d), dtype=torch.uint8, device="cuda")
                ts = []
                for i in range(args.warmup + args.steps):
                    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    e0.record()
                    F.fxpq_conv_fwd(d, x, w, b, y, ws=ws)
                    e1.record()
                    e1.synchronize()
                    if i >= args.warmup:
                        ts.append(e0.elapsed_time(e1))
                ms = sum(ts) / len(ts)
                wbytes = w.numel() * 2 if packed is None else packed.numel()
                out[name] = {"ms": round(ms, 4), "weight_bytes": wbytes, "weight_gbs": round(wbytes / (ms / 1e3) / 1e9, 1)}
    if args.kernel in ("config1", "all"):
        out.update(bench_config1(args, F))
    if args.kernel in ("config2", "all"):
        out.update(bench_config2(args, F))
    if args.kernel in ("forward", "all"):
        # the integer forward of the bench workload alone (one plan, calibrated once): the target of the
        # per-launch DRAM traffic capture of the conv kernels
        from paper_2203_12091_gb300.net import QNet
        wl = WORKLOADS[args.workload]
        arch, B = wl["arch"], wl["batch"]
        imgs = torch.from_numpy(synth.images(B, wl["seed"])).cuda()
        wdev, bndev = device_params(arch, wl["seed"], imgs.device)
        plan = synth.bit_plan(arch, wl["plans"][0])
        q = QNet(synth.ARCHS[arch](), hw=224, cin=3)
        q._dev = imgs.device
        q.quantize_params(wdev, plan, None, bndev)
        q.calibrate(imgs[: wl["calib"]], plan)
        out["memory"] = {k: round(v, 3) for k, v in q.memory().items()}
        ts = []
        for i in range(args.warmup + args.steps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            q.forward(imgs)
            e1.record()
            e1.synchronize()
            if i >= args.warmup:
                ts.append(e0.elapsed_time(e1))
        ms = sum(ts) / len(ts)
        out["forward"] = {"workload": args.workload, "ms": round(ms, 4), "images_s": round(B / (ms / 1e3), 1)}
    print(json.dumps({"kernel_timing": out}))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--kernel", choices=["conv", "flsearch", "quantize", "fopt", "forward", "fc", "config1", "config2",
                                         "all"],
                    help="time one kernel case and exit")
    ap.add_argument("--oracle-job", default=None, help=argparse.SUPPRESS)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="fxpq", choices=["fxpq", "reference"])
    ap.add_argument("--workload", default="vgg16", choices=sorted(WORKLOADS))
    ap.add_argument("--no-cpu", action="store_true", help="skip the oracle cpu_baseline leg")
    args = ap.parse_args()
    if args.oracle_job:
        oracle_job(args.oracle_job)
    elif args.kernel:
        run_kernel(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_fxpq(args)


if __name__ == "__main__":
    main()
