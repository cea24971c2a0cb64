"""Benchmark of the 1xN-pruned convolution forward pass on GB300.

Workload (one "step"): the ResNet-50 stage-2 3x3 convolution, batch 64,
28x28, 128 -> 128 channels, stride 1, pad 1, 1xN blocks with N = 8 at a 50%
block pruning rate, run once with fp32 inputs ("f32" leg) and once with bf16
inputs / fp32 accumulation ("bf16" leg).  Inputs are seeded synthetic
tensors resident in HBM; L2 is flushed (256 MB write) before every step.

Prints one JSON line.  Metric: effective TFLOP/s = 2 * pixels * t * N / time
(t = kept blocks), summed over both legs.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

--impl reference times the CPU oracle (fp64, plain C) on the host cores on a
bounded pixel sample of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

METRIC = "1xN sparse conv effective TFLOP/s and % of roofline; speedup vs own dense path"
L2_FLUSH_BYTES = 256 << 20
SM_COUNT_GB300 = 152
FP32_LANES_PER_SM = 128


def workload():
    from paper_2105_14713_gb300 import workloads as wl
    return [wl.config2("f32")[0], wl.config2("bf16")[0]]


def kept_flops(layer, t):
    return 2.0 * layer.pixels * t * layer.N


def alg_bytes(layer, t):
    """X + Y + D + I + P, each once (halo re-reads and skipped work not counted)."""
    es = 4 if layer.dtype == "f32" else 2
    x = layer.B * layer.H * layer.W * layer.C_in * es
    y = layer.pixels * layer.C_out * es
    return x + y + t * layer.N * es + t * 4 + (layer.C_out // layer.N + 1) * 4


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    src = "measured"
    try:
        with open(path) as fh:
            pk = json.load(fh)
        hbm, bf16 = float(pk["hbm_gbs"]), float(pk["bf16_tflops"])
        bf16_s = float(pk.get("bf16_tflops_sustained", bf16))
        sm_max = float(pk.get("sm_max_mhz", 2070.0))
    except (OSError, KeyError, ValueError):
        hbm, bf16, bf16_s, sm_max, src = 6800.0, 1900.0, 1700.0, 2070.0, "fallback"
    # FFMA peak: 152 SMs x 128 fp32 lanes x 2 flop x max SM clock.
    fp32 = SM_COUNT_GB300 * FP32_LANES_PER_SM * 2 * sm_max * 1e6 / 1e12
    return {"hbm_gbs": hbm, "bf16_tflops": bf16, "bf16_tflops_sustained": bf16_s,
            "fp32_ffma_tflops": fp32, "sm_max_mhz": sm_max, "source": src}


class ClockSampler:
    """nvidia-smi sampling of SM clock and throttle reasons during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = os.path.join("/tmp", f"onexn_clocks_{os.getpid()}.csv")

    def __enter__(self):
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "100"], stdout=self.fh,
                stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.fh.close()

    def summary(self):
        if self.proc is None:
            return None
        rows = []
        with open(self.path) as fh:
            for line in fh:
                f = [c.strip() for c in line.split(",")]
                if len(f) < 9:
                    continue
                try:
                    rows.append((float(f[1]), float(f[2]), f[5:9]))
                except ValueError:
                    continue
        try:
            os.unlink(self.path)
        except OSError:
            pass
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, fl in rows for i, v in enumerate(fl)
                          if v.lower() == "active"})
        smax = max(r[1] for r in rows)
        loaded = [r[0] for r in rows if r[0] > 0.5 * smax] or [r[0] for r in rows]
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": smax, "reasons": reasons,
                "samples": len(rows)}


def traffic_for(kernel_key: str):
    """DRAM bytes per launch from a committed ncu summary, only if the kernel
    source is unchanged since the counters were taken."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as fh:
            rec = json.load(fh).get(kernel_key)
    except (OSError, ValueError):
        return None
    if not rec:
        return None
    src = os.path.join(ROOT, rec["source"])
    try:
        sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    except OSError:
        return None
    return rec["dram_bytes_per_launch"] if sha == rec["source_sha"] else None


# --------------------------------------------------------------------------
# distributed plumbing (replicas: no data-path collective)
# --------------------------------------------------------------------------

def dist_setup(n_gpus: int):
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if ws > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend=backend)
    return rank, local, ws


def barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        if dist.get_backend() == "nccl":
            dist.barrier(device_ids=[torch.cuda.current_device()])
        else:
            dist.barrier()


def max_over_ranks(v: float, ws: int) -> float:
    if ws == 1:
        return v
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([v], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# --------------------------------------------------------------------------
# oracle (CPU baseline and the reference arm)
# --------------------------------------------------------------------------

def oracle_step(layers, packs, pixels):
    import oracle
    t0 = time.perf_counter()
    flops = 0.0
    for layer, (x, P, I, D, b) in zip(layers, packs):
        oracle.conv_bsr(x, P, I, D, layer.C_out, layer.KH, layer.KW, layer.N, b,
                        (layer.stride,) * 2, (layer.pad,) * 2, (layer.dil,) * 2, pixels=pixels)
        flops += 2.0 * len(pixels) * len(I) * layer.N
    return time.perf_counter() - t0, flops


def oracle_setup(layers):
    import oracle
    from paper_2105_14713_gb300 import workloads as wl
    packs = []
    for layer in layers:
        W = wl.weights(layer).numpy()
        x = wl.activations(layer).numpy()
        if layer.dtype == "bf16":
            x = oracle.round_bf16(x)
        mask, _ = oracle.prune(W, layer.N, layer.rate)
        P, I, D = oracle.pack(W, mask, layer.N, layer.dtype)
        packs.append((x, P, I, D, wl.bias(layer).numpy()))
    return packs


def cpu_baseline(layers, budget_s: float = 10.0):
    """The oracle as it stands, on this host's cores, on a bounded sample:
    whole images (784 output pixels each), as many as fit in ~budget_s."""
    import oracle
    packs = oracle_setup(layers)
    npix_img = layers[0].Ho * layers[0].Wo
    n_img, spent, flops = 0, 0.0, 0.0
    while spent < budget_s and n_img < layers[0].B:
        pix = np.arange(n_img * npix_img, (n_img + 1) * npix_img, dtype=np.int64)
        dt, fl = oracle_step(layers, packs, pix)
        spent += dt
        flops += fl
        n_img += 1
    return {"value": flops / spent / 1e12, "unit": "TFLOP/s", "cores": oracle.num_threads(),
            "kind": "oracle",
            "sample": f"{n_img} of {layers[0].B} images ({n_img * npix_img} output pixels x all "
                      f"{layers[0].C_out} channels), both legs, fp64 plain-C oracle, "
                      f"{spent:.1f} s"}


def run_reference(args, rank, ws):
    if rank != 0:
        return
    import oracle
    layers = workload()
    packs = oracle_setup(layers)
    npix_img = layers[0].Ho * layers[0].Wo
    rng = np.random.default_rng(0)
    times, flops = [], []
    for i in range(args.warmup + args.steps):
        img = int(rng.integers(0, layers[0].B))
        pix = np.arange(img * npix_img, (img + 1) * npix_img, dtype=np.int64)
        dt, fl = oracle_step(layers, packs, pix)
        if i >= args.warmup:
            times.append(dt)
            flops.append(fl)
    v = sum(flops) / sum(times) / 1e12
    ms = 1e3 * sum(times) / len(times)
    sample = (f"one random image per step (784 output pixels x 128 channels), both legs; "
              f"fp64 plain-C oracle, {oracle.num_threads()} threads")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": v, "unit": "TFLOP/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": config_json(layers, "cpu oracle sample"),
        "cpu_baseline": {"value": v, "unit": "TFLOP/s", "cores": oracle.num_threads(),
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": v, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


def config_json(layers, l2="flushed before every step (256 MB write)"):
    l0 = layers[0]
    return {"workload": "ResNet-50 stage-2 3x3 conv, 64x28x28x128 -> 128, s1 p1, NHWC; "
                        "1xN N=8, 50% block rate; fp32 leg + bf16-in/fp32-acc leg",
            "batch": l0.B, "H": l0.H, "W": l0.W, "C_in": l0.C_in, "C_out": l0.C_out,
            "kernel": [l0.KH, l0.KW], "N": l0.N, "rate": l0.rate,
            "legs": [l.dtype for l in layers], "parallelism": "replicas", "l2": l2}


# --------------------------------------------------------------------------
# GPU arm
# --------------------------------------------------------------------------

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    rank, local, ws = dist_setup(args.gpus)
    if args.impl == "reference":
        run_reference(args, rank, ws)
        return

    from paper_2105_14713_gb300 import onexn as ox
    from paper_2105_14713_gb300 import workloads as wl
    from paper_2105_14713_gb300.layer import PrunedConv2d

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    layers = workload()
    legs = []
    for layer in layers:
        W = wl.weights(layer).numpy()
        conv = PrunedConv2d(W, layer.N, layer.rate, bias=wl.bias(layer).numpy(),
                            stride=layer.stride, padding=layer.pad, dilation=layer.dil,
                            dtype=layer.dtype, device=dev)
        x_cpu = wl.activations(layer)
        x_cpu = x_cpu if layer.dtype == "f32" else x_cpu.to(torch.bfloat16)
        x = x_cpu.to(dev)
        y = torch.empty(conv.out_shape(x.shape), dtype=x.dtype, device=dev)
        legs.append({"layer": layer, "conv": conv, "x": x, "y": y,
                     "x_host": x_cpu.pin_memory(), "algo": conv.algo(x.shape)})
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)

    def step(evs=None):
        for i, lg in enumerate(legs):
            if evs is not None:
                evs[i][0].record(stream)
            lg["conv"](lg["x"], lg["y"])
            if evs is not None:
                evs[i][1].record(stream)

    for _ in range(args.warmup):
        flush.fill_(1)
        step()
    torch.cuda.synchronize()

    # ---- timed region: K steps, L2 flushed before each (outside the events) ----
    evs = [[[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in legs]
           for _ in range(args.steps)]
    sampler = ClockSampler(local)
    barrier(ws)
    torch.cuda.synchronize()
    with sampler:
        wall0 = time.perf_counter()
        for k in range(args.steps):
            flush.fill_(k & 0xff)
            step(evs[k])
        torch.cuda.synchronize()
        wall = time.perf_counter() - wall0
    barrier(ws)
    leg_ms = [[evs[k][i][0].elapsed_time(evs[k][i][1]) for k in range(args.steps)]
              for i in range(len(legs))]
    step_ms = sum(sum(m) for m in leg_ms) / args.steps
    step_ms_max = max_over_ranks(step_ms, ws)
    flops_step = sum(kept_flops(lg["layer"], lg["conv"].t) for lg in legs)
    value = ws * flops_step / (step_ms_max * 1e-3) / 1e12
    clocks = sampler.summary()

    # ---- per-leg roofline (live CUDA-event durations of each kernel) ----
    pk = peaks()
    leg_info = []
    for i, lg in enumerate(legs):
        layer, t = lg["layer"], lg["conv"].t
        ms = sum(leg_ms[i]) / len(leg_ms[i])
        fl, by = kept_flops(layer, t), alg_bytes(layer, t)
        if lg["algo"] == "fma":
            bound_peak, unit_peak, bound = pk["fp32_ffma_tflops"], "TFLOP/s", "alu"
        else:
            bound_peak, unit_peak, bound = pk["bf16_tflops"], "TFLOP/s", "tensor"
        t_roof = max(fl / (bound_peak * 1e12), by / (pk["hbm_gbs"] * 1e9))
        leg_info.append({
            "dtype": layer.dtype, "algo": lg["algo"], "ms": ms, "t_kept_blocks": t,
            "tflops": fl / (ms * 1e-3) / 1e12, "gbs": by / (ms * 1e-3) / 1e9,
            "roofline_frac": t_roof / (ms * 1e-3), "bound": bound,
            "pipe_peak_tflops": bound_peak})

    dom = max(range(len(legs)), key=lambda i: leg_info[i]["ms"])
    dl = leg_info[dom]
    dlay = legs[dom]["layer"]
    roof = {"bound": dl["bound"], "achieved": dl["tflops"], "peak": dl["pipe_peak_tflops"],
            "unit": "TFLOP/s", "frac": dl["tflops"] / dl["pipe_peak_tflops"],
            "traffic": traffic_for(f"{dl['algo']}_{dlay.dtype}_cfg2"),
            "kernel": f"{dl['algo']} ({dlay.dtype} leg)",
            "peak_source": ("FFMA: 152 SMs x 128 lanes x 2 x %.0f MHz (derived)" % pk["sm_max_mhz"]
                            if dl["bound"] == "alu" else f"{pk['source']} bf16 tensor")}

    # ---- dense path (rate 0, N = C_out) at the same shape, same timing method ----
    speedup = {}
    for lg in legs:
        layer = lg["layer"]
        dl_layer = wl.dense_counterpart(layer)
        dconv = PrunedConv2d(wl.weights(layer).numpy(), dl_layer.N, 0.0,
                             bias=wl.bias(layer).numpy(), stride=layer.stride,
                             padding=layer.pad, dilation=layer.dil, dtype=layer.dtype,
                             device=dev)
        dts = []
        for r in range(args.warmup + 10):
            flush.fill_(r & 0xff)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            dconv(lg["x"], lg["y"])
            e1.record(stream)
            torch.cuda.synchronize()
            if r >= args.warmup:
                dts.append(e0.elapsed_time(e1))
        dense_ms = sum(dts) / len(dts)
        sparse_ms = [li for li in leg_info if li["dtype"] == layer.dtype][0]["ms"]
        speedup[layer.dtype] = {"dense_ms": dense_ms, "sparse_ms": sparse_ms,
                                "speedup": dense_ms / sparse_ms,
                                "dense_algo": dconv.algo(lg["x"].shape)}

    # ---- end to end through the public API, host buffers, copies timed ----
    e2e_ms = []
    h2d = sum(lg["x_host"].numel() * lg["x_host"].element_size() for lg in legs)
    d2h = sum(lg["y"].numel() * lg["y"].element_size() for lg in legs)
    y_host = [torch.empty(lg["y"].shape, dtype=lg["y"].dtype, pin_memory=True) for lg in legs]
    for r in range(args.warmup + args.steps):
        flush.fill_(r & 0xff)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i, lg in enumerate(legs):
            xd = lg["x_host"].to(dev, non_blocking=True)
            yd = lg["conv"](xd)
            y_host[i].copy_(yd, non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize()
        if r >= args.warmup:
            e2e_ms.append(e0.elapsed_time(e1))
    e2e_step = max_over_ranks(sum(e2e_ms) / len(e2e_ms), ws)

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(layers)

    if rank == 0:
        out = {
            "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": step_ms_max,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f32+bf16", "data": "synthetic (seeded Kaiming-normal weights, ReLU(N(0,1)) "
                                         "activations)",
            "config": config_json(layers),
            "roofline": roof,
            "legs": leg_info,
            "speedup_vs_dense": speedup,
            "e2e": {"value": ws * flops_step / (e2e_step * 1e-3) / 1e12, "unit": "TFLOP/s",
                    "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "ms_per_step": e2e_step},
            "gpu_launches": len(legs) * args.steps,
            "clocks": clocks,
            "wall_s_timed_region": wall,
            "peaks": pk,
            "cpu_baseline": cpu,
        }
        print(json.dumps(out), flush=True)
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
