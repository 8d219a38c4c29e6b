"""Benchmark of the per-channel quantized linear (OutlierTune, arXiv 2406.18832)
on GB300.

Headline workload: the OPT-66B-shaped FFN linears (fc1 9216->36864, fc2
36864->9216) at a prefill of 4096 tokens, W8A8, with synthetic LayerNorm-like
activations carrying 1% fixed outlier channels (x U[30, 100], offsets
U[-40, 40]).  Offline per layer (not in the step, measured separately):
calibration over 65,536 tokens and the weight fold.  One step = for each of
the two layers, the symmetrize+quantize kernel then the tcgen05 GEMM with its
fused epilogue.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Prints one JSON line.  The value is exact int8 tera-operations per second
(2*M*N*K per linear) over the whole step.  Beside it: the OPT-6.7B step at
2048 tokens, the OPT-30B block, decode-sized and swept token counts (each
against cuBLAS fp16 of the same shapes), the fused LayerNorm, the per-token
path, asymmetric weights and the clipping calibration.  --impl reference
times the CPU oracle on a bounded sample of the headline workload on the host
cores.
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
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

WORKLOAD_CFG = 4          # OPT-66B-shaped fc1 / fc2
WORKLOAD_NAME = "opt-66b-ffn-prefill-4096"
TOKENS = 4096
BITS = (8, 8)
STEP6_CFG, STEP6_TOKENS = 2, 2048   # the OPT-6.7B step beside the headline
METRIC = "W8A8 linear TOPS & % INT8 peak; quantize GB/s % HBM; vs cuBLAS FP16"
L2_BYTES = 129 * 2 ** 20


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return dict(hbm=float(p["hbm_gbs"]), bf16=float(p["bf16_tflops"]),
                    bf16_sus=float(p["bf16_tflops_sustained"]), source="measured")
    except Exception:
        return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, source="fallback")


def _env_rank():
    return int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")), \
        int(os.environ.get("LOCAL_RANK", "0"))


def _workload_desc(cfg: int = WORKLOAD_CFG):
    from paper_2406_18832_gb300 import synth
    c = synth.CONFIGS[cfg]
    return c, [(l.name, l.K, l.N) for l in c.layers]


def _ops_per_step(layers, tokens):
    return sum(2 * tokens * K * N for _, K, N in layers)


def max_over_ranks(value: float, device=None) -> float:
    """Largest `value` over all ranks (the job is as slow as its slowest replica)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(ops_per_rank_step: int, world: int, steps: int, max_ms: float) -> float:
    """Whole-job throughput in tera-ops/s: every replica runs the full workload
    (weak scaling), so the units of all ranks divide by the slowest rank's time."""
    return world * ops_per_rank_step * steps / (max_ms * 1e-3) / 1e12


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""

    FIELDS = "index,clocks.sm,clocks.max.sm,power.draw.instant,clocks_event_reasons.active," \
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown," \
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap"

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "20"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *a):
        self.out = ""
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = []
        for line in (self.out or "").strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append(dict(sm=float(parts[1]), max=float(parts[2]), power=float(parts[3]),
                                 hw=parts[5], hwt=parts[6], swt=parts[7], pcap=parts[8]))
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        loaded = [r for r in rows if r["power"] > 200.0] or rows
        reasons = set()
        for r in loaded:
            for key, name in (("hw", "hw_slowdown"), ("hwt", "hw_thermal_slowdown"),
                              ("swt", "sw_thermal_slowdown"), ("pcap", "sw_power_cap")):
                if r[key].lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(r["sm"] for r in loaded), "sm_max_mhz": max(r["max"] for r in rows),
                "reasons": sorted(reasons), "samples": len(loaded),
                "power_w_max": max(r["power"] for r in rows)}


def _traffic_record():
    """DRAM bytes per GEMM launch of the headline workload from the committed
    ncu summary, if the GEMM source is unchanged since it was captured and the
    summary is of this workload (else None)."""
    path = os.path.join(ROOT, "profiles", "linear_pair_kernel_traffic_opt66b_ffn_m4096.txt")
    src = os.path.join(ROOT, "paper_2406_18832_gb300", "csrc", "gemm.cu")
    try:
        sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        vals = {}
        for line in open(path):
            line = line.strip()
            if "=" in line and not line.startswith("#"):
                k, v = line.split("=", 1)
                vals[k.strip()] = v.strip()
        if vals.get("gemm_cu_sha256_16") != sha or vals.get("workload") != WORKLOAD_NAME:
            return None
        return float(vals["dram_bytes_per_launch"])
    except Exception:
        return None


# ----------------------------------------------------------------------------
# the CUDA path
# ----------------------------------------------------------------------------
def _build_layers(dev, cfg_index, tokens, bits, t_cal=None):
    """Calibrated and folded QuantizedLinear per layer of a config, with its
    runtime activations; calibration and fold are timed (offline steps)."""
    import torch

    from paper_2406_18832_gb300 import QuantizedLinear, synth
    cfg = synth.CONFIGS[cfg_index]
    bits_a, bits_w = bits
    layers, xs = [], []
    calib_ms, calib_bytes, fold_ms = [], 0, []
    for li, layer in enumerate(cfg.layers):
        w, b = synth.weights(cfg_index, li, layer, device=dev)
        xc = synth.activations(cfg_index, li, layer, t_cal or cfg.T_cal, 3, device=dev)
        x = synth.activations(cfg_index, li, layer, tokens, 4, device=dev)
        ql = QuantizedLinear(layer.K, layer.N, bits_a, bits_w, relu=layer.relu_out, device=dev)
        # calibration: warm once, then time one pass over the calibration tokens
        ql.calibrate(xc)
        ql._calibrated = False
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        ql.calibrate(xc)
        e1.record()
        torch.cuda.synchronize()
        calib_ms.append(e0.elapsed_time(e1))
        calib_bytes += xc.numel() * 2
        e0.record()
        ql.fold(w, b)
        e1.record()
        torch.cuda.synchronize()
        fold_ms.append(e0.elapsed_time(e1))
        del xc
        layers.append((ql, w, b))
        xs.append(x)
    torch.cuda.empty_cache()
    return layers, xs, calib_ms, calib_bytes, fold_ms


def _timed_steps(layers, xs, qbufs, ybufs, steps, stream):
    """Run `steps` steps (quantize then linear per layer) with CUDA events
    around every launch; returns total ms and per-layer lists of GEMM and
    quantize ms."""
    import torch
    nl = len(layers)
    events = [[[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(nl)] for _ in range(steps)]
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for k in range(steps):
        for i, (ql, _, _) in enumerate(layers):
            events[k][i][0].record(stream)
            ql.quantize(xs[i], qbufs[i])
            events[k][i][1].record(stream)
            ql.linear(qbufs[i], ybufs[i])
            events[k][i][2].record(stream)
    t1.record(stream)
    torch.cuda.synchronize()
    gemm_ms = [[events[k][i][1].elapsed_time(events[k][i][2]) for k in range(steps)] for i in range(nl)]
    quant_ms = [[events[k][i][0].elapsed_time(events[k][i][1]) for k in range(steps)] for i in range(nl)]
    return t0.elapsed_time(t1), gemm_ms, quant_ms


def _cublas_ms(xs, ws, ybufs, reps):
    """cuBLAS fp16 GEMM (torch.matmul) of each layer's shape, ms per call."""
    import torch
    out = []
    for x, w, y in zip(xs, ws, ybufs):
        def f():
            torch.matmul(x, w.t(), out=y)
        for _ in range(3):
            f()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            f()
        e1.record()
        torch.cuda.synchronize()
        out.append(e0.elapsed_time(e1) / reps)
    return out


def _quant_stats(layer_shapes, tokens, quant_ms, steps):
    """Quantize throughput on the algorithmic bytes (fp16 X in, int8 codes
    out, z and r) and on the bytes the kernel moves (fp16 codes out)."""
    alg = sum(3 * tokens * K + 8 * K for _, K, _ in layer_shapes)
    moved = sum(4 * tokens * K + 8 * K for _, K, _ in layer_shapes)
    t = sum(sum(v) for v in quant_ms) / steps
    return alg, moved, t


def run_ours(args):
    import torch
    import torch.distributed as dist

    from paper_2406_18832_gb300 import binding

    rank, world, local = _env_rank()
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    binding.load()
    peaks = _peaks()
    cfg, layer_shapes = _workload_desc()
    bits_a, bits_w = BITS

    if args.profile_opt67b:
        # profiler runs of the OPT-6.7B step (QKV, out, fc1, fc2 at 2048 tokens, W8A8): quantize then
        # linear per layer, `warmup` + `steps` steps, nothing else
        layers, xs, _, _, _ = _build_layers(dev, STEP6_CFG, STEP6_TOKENS, BITS, 8192)
        c6 = _workload_desc(STEP6_CFG)[0]
        qb = [torch.empty(STEP6_TOKENS, l.K, dtype=torch.float16, device=dev) for l in c6.layers]
        yb = [torch.empty(STEP6_TOKENS, l.N, dtype=torch.float16, device=dev) for l in c6.layers]
        for _ in range(args.warmup + args.steps):
            for i, (ql, _, _) in enumerate(layers):
                ql.forward(xs[i], qb[i], yb[i])
        torch.cuda.synchronize()
        if rank == 0:
            print(json.dumps({"profile_run": "opt67b", "steps": args.steps, "warmup": args.warmup}), flush=True)
        return

    if args.profile_decode or args.profile_linear:
        # profiler runs of the decode- / mid-sized linears only: nothing else is set up
        tokens = args.profile_linear or 0
        res = bench_decode(dev, peaks, reps=args.steps) if args.profile_decode else \
            profile_linears(dev, tokens, args.steps, args.warmup)
        torch.cuda.synchronize()
        if rank == 0:
            print(json.dumps({"profile_run": "decode" if args.profile_decode else f"linear-{tokens}",
                              "steps": args.steps, "result": res}), flush=True)
        return

    # ---- offline: inputs, calibration, fold (each rank its own replica) ----
    layers, xs, calib_ms, calib_bytes, fold_ms = _build_layers(dev, WORKLOAD_CFG, TOKENS, BITS,
                                                               8192 if args.profile else None)
    qbufs = [torch.empty(TOKENS, l.K, dtype=torch.float16, device=dev) for l in cfg.layers]
    ybufs = [torch.empty(TOKENS, l.N, dtype=torch.float16, device=dev) for l in cfg.layers]
    ops_step = _ops_per_step(layer_shapes, TOKENS)
    stream = torch.cuda.current_stream()

    def step():
        for i, (ql, _, _) in enumerate(layers):
            ql.quantize(xs[i], qbufs[i])
            ql.linear(qbufs[i], ybufs[i])

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()

    if args.profile:
        # small, short run for profilers: the steps only, nothing else
        for _ in range(args.steps):
            step()
        torch.cuda.synchronize()
        if rank == 0:
            print(json.dumps({"profile_run": True, "steps": args.steps}), flush=True)
        return

    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(torch.cuda.current_device() if world == 1 else local) as clk:
        total_ms, gemm_ms, quant_ms = _timed_steps(layers, xs, qbufs, ybufs, args.steps, stream)
    if world > 1:
        dist.barrier()
    total_ms = max_over_ranks(total_ms, dev)
    ms_per_step = total_ms / args.steps
    value = job_value(ops_step, world, args.steps, total_ms)

    # GEMM roofline (dominant kernel): algorithmic ops / measured launch time
    gemm_ops = [2 * TOKENS * K * N for _, K, N in layer_shapes]
    gemm_time = sum(sum(v) for v in gemm_ms)
    gemm_tops = sum(o * args.steps for o in gemm_ops) / (gemm_time * 1e-3) / 1e12
    cub = _cublas_ms(xs, [w for _, w, _ in layers], ybufs, max(5, min(50, args.steps)))
    per_layer = []
    for i, (name, K, N) in enumerate(layer_shapes):
        g = statistics.median(gemm_ms[i])
        q = statistics.median(quant_ms[i])
        per_layer.append({"layer": name, "K": K, "N": N, "gemm_us": round(g * 1e3, 2),
                          "gemm_tops": round(gemm_ops[i] / (g * 1e-3) / 1e12, 1),
                          "gemm_frac_peak": round(gemm_ops[i] / (g * 1e-3) / 1e12 / peaks["bf16"], 4),
                          "cublas_fp16_us": round(cub[i] * 1e3, 2),
                          "cublas_fp16_tflops": round(gemm_ops[i] / (cub[i] * 1e-3) / 1e12, 1),
                          "quant_us": round(q * 1e3, 2),
                          "quant_gbs_algorithmic": round((3 * TOKENS * K + 8 * K) / (q * 1e-3) / 1e9, 1),
                          "quant_gbs_moved": round((4 * TOKENS * K + 8 * K) / (q * 1e-3) / 1e9, 1)})
    q_alg, q_moved, quant_time = _quant_stats(layer_shapes, TOKENS, quant_ms, args.steps)
    clocks = clk.summary()
    long_run = total_ms > 4000.0
    peak = peaks["bf16_sus"] if long_run else peaks["bf16"]
    roofline = {"kernel": "linear_pair_kernel (tcgen05 cta_group::2 kind::f16, exact int8 codes)", "bound": "tensor",
                "achieved": round(gemm_tops, 1), "peak": peak, "unit": "TFLOP/s",
                "frac": round(gemm_tops / peak, 4), "traffic": _traffic_record(),
                "peak_source": f"{peaks['source']} bf16 dense {'sustained' if long_run else 'burst'} "
                               "(fp16 dense runs at the bf16 rate)",
                "algorithmic": "2 M N K ops per launch (M = 4096; fc1 and fc2: 2.78 T each)"}

    int8_tops = None
    try:
        _, K0, N0 = layer_shapes[0]
        a8 = torch.randint(-127, 128, (TOKENS, K0), device=dev, dtype=torch.int8)
        b8 = torch.randint(-127, 128, (K0, N0), device=dev, dtype=torch.int8)
        for _ in range(2):
            torch._int_mm(a8, b8)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(3):
            torch._int_mm(a8, b8)
        e1.record()
        torch.cuda.synchronize()
        int8_tops = 2 * TOKENS * K0 * N0 / (e0.elapsed_time(e1) / 3 * 1e-3) / 1e12
        del a8, b8
    except Exception:
        int8_tops = None

    # ---- end to end through the public API, host buffers in and out ----
    e2e_steps = max(3, min(50, args.steps))
    e2e_ms, h2d, d2h = _e2e(layers, xs, qbufs, ybufs, e2e_steps)

    # ---- host copies for the CPU oracle baseline (rank 0, one replica) ----
    host = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        host = [dict(w=w.cpu().numpy(), b=b.cpu().numpy(), x=x[:1024].cpu().numpy(), relu=ql.relu,
                     xc=None) for (ql, w, b), x in zip(layers, xs)]
        from paper_2406_18832_gb300 import synth
        for li, layer in enumerate(cfg.layers):
            host[li]["xc"] = synth.activations(WORKLOAD_CFG, li, layer, 8192, 3, device=dev).cpu().numpy()

    weights_fp16 = sum(2 * K * N for _, K, N in layer_shapes)
    weights_int8 = sum(ql.weight_bytes() for ql, _, _ in layers)
    del layers, xs, qbufs, ybufs
    torch.cuda.empty_cache()

    def fresh():
        # each stage allocates its tensors anew rather than from blocks the
        # caching allocator kept from earlier, larger stages (measured: a
        # decode point drawn from such blocks ran 15-25 % slow in one run of
        # three, in the same place each time; fresh allocations did not)
        torch.cuda.synchronize()
        torch.cuda.empty_cache()

    step6 = bench_step6(dev, peaks, max(5, min(200, args.steps)), args.warmup)
    fresh()
    block = None if args.no_block else bench_block(dev)
    fresh()
    decode = bench_decode(dev, peaks)
    fresh()
    lnq = bench_layernorm(dev, peaks)
    fresh()
    qsweep = bench_quantize_sweep(dev, peaks)
    fresh()
    sweep = bench_token_sweep(dev, peaks)
    fresh()
    per_tok = bench_per_token(dev, peaks)
    fresh()
    clip = bench_clipping(dev, peaks, step6.pop("_calib_ms0"))

    cpu = None
    if host is not None:
        cpu = cpu_baseline(host, budget_s=args.cpu_budget)

    line = {
        "metric": METRIC, "value": round(value, 2), "unit": "TOPS", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms_per_step, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None,
        "dtype": "int8 codes exact on the f16 tensor pipe (fp32 chunk sums, int32 totals)",
        "data": "synthetic",
        "config": {"workload": WORKLOAD_NAME, "tokens": TOKENS, "bits_a": bits_a, "bits_w": bits_w,
                   "layers": [{"name": n, "K": K, "N": N} for n, K, N in layer_shapes],
                   "calibration_tokens": cfg.T_cal, "parallelism": f"replicas x{world}",
                   "l2": "inputs larger than L2: one step streams 680 MB of int8 weights and 1.3 GB of "
                         "activations, codes and outputs through the 129 MB L2"},
        "roofline": roofline,
        "gpu_launches": args.steps * 2 * len(layer_shapes),
        "e2e": {"value": round(ops_step / (e2e_ms * 1e-3) / 1e12 * world, 2), "unit": "TOPS",
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": round(e2e_ms, 4),
                "copies": "pinned host buffers; host->device, layers and device->host on three streams, buffers alternating between two sets from step to step"},
        "clocks": clocks,
        "quantize": {"gbs_algorithmic": round(q_alg / (quant_time * 1e-3) / 1e9, 1),
                     "frac_algorithmic": round(q_alg / (quant_time * 1e-3) / 1e9 / peaks["hbm"], 4),
                     "gbs_moved": round(q_moved / (quant_time * 1e-3) / 1e9, 1),
                     "frac_moved": round(q_moved / (quant_time * 1e-3) / 1e9 / peaks["hbm"], 4),
                     "hbm_peak_gbs": peaks["hbm"], "bytes_algorithmic_per_step": q_alg,
                     "bytes_moved_per_step": q_moved,
                     "note": "algorithmic: fp16 X in + int8 codes out + z, r; moved: the fp16 codes the "
                             "prefill GEMM reads", "sweep": qsweep},
        "calibrate": {"gbs": round(calib_bytes / (sum(calib_ms) * 1e-3) / 1e9, 1),
                      "frac": round(calib_bytes / (sum(calib_ms) * 1e-3) / 1e9 / peaks["hbm"], 4),
                      "tokens": cfg.T_cal, "ms_per_layer": [round(v, 3) for v in calib_ms]},
        "fold_ms_per_layer": [round(v, 3) for v in fold_ms],
        "cublas_fp16": {"ms_per_step": round(sum(cub), 4),
                        "tflops": round(ops_step / (sum(cub) * 1e-3) / 1e12, 1),
                        "ours_over_cublas": round(sum(cub) / ms_per_step, 4),
                        "gemm_only_over_cublas": round(sum(cub) / (gemm_time / args.steps), 4)},
        "int8_peak": {"cublaslt_int8_tops": None if int8_tops is None else round(int8_tops, 1),
                      "frac_of_cublaslt_int8": None if not int8_tops else round(gemm_tops / int8_tops, 2),
                      "note": "GB300 (sm_103a) has no tcgen05 int8 MMA; cuBLASLt int8 (torch._int_mm) of the "
                              "fc1 shape, measured in this run"},
        "per_layer": per_layer,
        "memory": {"weights_fp16_bytes": weights_fp16, "weights_int8_bytes": weights_int8,
                   "ratio": round(weights_fp16 / weights_int8, 3)},
        "opt67b_step": step6,
        "block": block,
        "decode": decode,
        "token_sweep": sweep,
        "per_token": per_tok,
        "layernorm_quantize": lnq,
        "clipping_calibration": clip,
        "cpu_baseline": cpu,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def _e2e(layers, xs, qbufs, ybufs, steps):
    """ms per step through the public API (QuantizedLinear.forward) with the
    inputs copied in from pinned host memory and the outputs copied back, as
    a pipelined server runs it: the copies go on their own streams, and the
    device inputs, device outputs and host outputs alternate between two sets
    from step to step, so a layer's input copy overlaps the layers before it,
    its output copy the layers after it, and no layer waits for the previous
    step's copy of the same buffer.  Every step's copies are inside the timed
    region."""
    import torch
    nb = 2
    hx = [x.cpu().pin_memory() for x in xs]
    hy = [[torch.empty(y.shape, dtype=y.dtype).pin_memory() for y in ybufs] for _ in range(nb)]
    dx = [[torch.empty_like(x) for x in xs] for _ in range(nb)]
    dy = [ybufs] + [[torch.empty_like(y) for y in ybufs] for _ in range(nb - 1)]
    s_c = torch.cuda.current_stream()
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    ev = [[[torch.cuda.Event() for _ in layers] for _ in range(nb)] for _ in range(3)]
    ev_in, ev_done, ev_out = ev

    def e2e_step(k):
        b = k % nb
        for i, (ql, _, _) in enumerate(layers):
            with torch.cuda.stream(s_in):
                s_in.wait_event(ev_done[b][i])       # the layer two steps back has read dx[b][i]
                dx[b][i].copy_(hx[i], non_blocking=True)
                ev_in[b][i].record(s_in)
            s_c.wait_event(ev_in[b][i])
            s_c.wait_event(ev_out[b][i])             # dy[b][i] of two steps back is copied out
            ql.forward(dx[b][i], qbufs[i], dy[b][i])
            ev_done[b][i].record(s_c)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev_done[b][i])
                hy[b][i].copy_(dy[b][i], non_blocking=True)
                ev_out[b][i].record(s_out)
    for k in range(2 * nb):
        e2e_step(k)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(s_c)
    s_in.wait_event(e0)
    s_out.wait_event(e0)
    for k in range(steps):
        e2e_step(k)
    s_c.wait_stream(s_in)
    s_c.wait_stream(s_out)
    e1.record(s_c)
    torch.cuda.synchronize()
    h2d = sum(x.numel() * 2 for x in xs)
    d2h = sum(y.numel() * 2 for y in ybufs)
    return e0.elapsed_time(e1) / steps, h2d, d2h


def bench_step6(dev, peaks, steps, warmup):
    """The OPT-6.7B step (QKV, out, fc1, fc2 at 2048 tokens, W8A8): quantize
    then linear per layer, as the headline; with the same step on the paper's
    "Int8" weights (per-output-channel zero points) beside it."""
    import torch
    cfg, shapes = _workload_desc(STEP6_CFG)
    layers, xs, calib_ms, calib_bytes, _ = _build_layers(dev, STEP6_CFG, STEP6_TOKENS, BITS)
    qbufs = [torch.empty(STEP6_TOKENS, l.K, dtype=torch.float16, device=dev) for l in cfg.layers]
    ybufs = [torch.empty(STEP6_TOKENS, l.N, dtype=torch.float16, device=dev) for l in cfg.layers]
    stream = torch.cuda.current_stream()
    for _ in range(warmup):
        for i, (ql, _, _) in enumerate(layers):
            ql.forward(xs[i], qbufs[i], ybufs[i])
    torch.cuda.synchronize()
    total_ms, gemm_ms, quant_ms = _timed_steps(layers, xs, qbufs, ybufs, steps, stream)
    ops_step = _ops_per_step(shapes, STEP6_TOKENS)
    ms = total_ms / steps
    gemm_ops = [2 * STEP6_TOKENS * K * N for _, K, N in shapes]
    gemm_tops = sum(o * steps for o in gemm_ops) / (sum(sum(v) for v in gemm_ms) * 1e-3) / 1e12
    cub = _cublas_ms(xs, [w for _, w, _ in layers], ybufs, 50)
    q_alg, q_moved, qt = _quant_stats(shapes, STEP6_TOKENS, quant_ms, steps)
    asym = bench_asym(dev, layers, xs, ops_step, ms)
    out = {"workload": "opt-6.7b-linears-prefill-2048", "tokens": STEP6_TOKENS, "ms_per_step": round(ms, 4),
           "tops": round(ops_step / (ms * 1e-3) / 1e12, 1), "gemm_tflops": round(gemm_tops, 1),
           "gemm_frac_peak": round(gemm_tops / peaks["bf16"], 4),
           "per_layer_gemm_us": [round(statistics.median(v) * 1e3, 2) for v in gemm_ms],
           "quantize_gbs_algorithmic": round(q_alg / (qt * 1e-3) / 1e9, 1),
           "cublas_fp16_ms_per_step": round(sum(cub), 4),
           "ours_over_cublas": round(sum(cub) / ms, 4), "asym_weights": asym,
           "_calib_ms0": (calib_ms[0], STEP6_CFG)}
    del layers, xs, qbufs, ybufs
    torch.cuda.empty_cache()
    return out


def bench_asym(dev, layers, xs, ops_step, ms_sym, reps: int = 200, t_cal: int = 8192):
    """The same OPT-6.7B prefill step with the paper's "Int8" weights
    (per-output-channel zero points): quantize with code row sums, then the
    linear whose epilogue subtracts zc_n * rowsum_m.  Calibrated on 8192
    tokens of the same synthetic stream as the main line."""
    import torch

    from paper_2406_18832_gb300 import QuantizedLinear, synth
    cfg = synth.CONFIGS[STEP6_CFG]
    qls = []
    for li, (layer, (ql_sym, w, b)) in enumerate(zip(cfg.layers, layers)):
        ql = QuantizedLinear(layer.K, layer.N, ql_sym.bits_a, ql_sym.bits_w, relu=layer.relu_out, device=dev,
                             weights="asym")
        ql.calibrate(synth.activations(STEP6_CFG, li, layer, t_cal, 3, device=dev)).fold(w, b)
        qls.append(ql)
    qb = [torch.empty(STEP6_TOKENS, ql.K, dtype=torch.float16, device=dev) for ql in qls]
    rb = [torch.empty(STEP6_TOKENS, dtype=torch.int32, device=dev) for _ in qls]
    yb = [torch.empty(STEP6_TOKENS, ql.N, dtype=torch.float16, device=dev) for ql in qls]
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in qls]
    gemm_ms = [0.0] * len(qls)

    def step(timed=False):
        for i, ql in enumerate(qls):
            if timed:
                evs[i][0].record()
            ql.quantize_with_rowsum(xs[i], qb[i], rb[i])
            if timed:
                evs[i][1].record()
            ql.linear(qb[i], yb[i], rowsum=rb[i])
            if timed:
                evs[i][2].record()

    for _ in range(5):
        step()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        step()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    for _ in range(20):
        step(timed=True)
        torch.cuda.synchronize()
        for i in range(len(qls)):
            gemm_ms[i] += evs[i][1].elapsed_time(evs[i][2]) / 20
    return {"workload": "opt-6.7b-linears-prefill, Int8 weights with zero points", "tokens": STEP6_TOKENS,
            "ms_per_step": round(ms, 4), "tops": round(ops_step / (ms * 1e-3) / 1e12, 1),
            "over_symmetric_step": round(ms / ms_sym, 4),
            "gemm_us_per_layer": [round(v * 1e3, 2) for v in gemm_ms]}


def profile_linears(dev, tokens: int, steps: int, warmup: int):
    """For profilers: `warmup` then `steps` eager calls of ot_linear on the
    OPT-13B QKV and fc2 shapes (Int6 codes and weights drawn directly) at
    `tokens` tokens, QKV then fc2 in each step."""
    import torch

    from paper_2406_18832_gb300 import binding, synth
    c = synth.CONFIGS[3]
    ws = torch.zeros(binding.ot_linear_workspace_size(), dtype=torch.uint8, device=dev)
    g = torch.Generator(device=dev).manual_seed(4100)
    args = []
    for li in (0, 3):
        N, K = c.layers[li].N, c.layers[li].K
        qw = torch.randint(-31, 32, (N, K), generator=g, device=dev, dtype=torch.int32).to(torch.int8)
        q = torch.randint(-31, 32, (tokens, K), generator=g, device=dev, dtype=torch.int32).half()
        args.append((q, qw, torch.rand(N, generator=g, device=dev) * 1e-3, torch.zeros(N, device=dev),
                     torch.empty(tokens, N, dtype=torch.float16, device=dev)))
    for k in range(warmup + steps):
        for q, qw, sw, bf, y in args:
            binding.ot_linear(q, qw, sw, bf, 6, 6, y, workspace=ws)
    torch.cuda.synchronize()
    return {"tokens": tokens, "layers": ["qkv 5120->15360", "fc2 20480->5120"], "calls": 2 * (warmup + steps)}


def bench_token_sweep(dev, peaks, reps: int = 20):
    """OPT-13B QKV and fc2 (Int6) at 1, 16, 128, 1024 and 4096 tokens: the
    linear alone (codes resident, consecutive calls on rotating weight copies
    so that weights come from HBM), CUDA-graph replay.  The roofline time of a
    point is the larger of its weight bytes over the HBM peak and its
    operations over the dense tensor peak; frac = roofline time / time."""
    import torch

    from paper_2406_18832_gb300 import binding, synth
    c = synth.CONFIGS[3]
    ws = torch.zeros(binding.ot_linear_workspace_size(), dtype=torch.uint8, device=dev)
    out = []
    for li in (0, 3):
        layer = c.layers[li]
        N, K = layer.N, layer.K
        g = torch.Generator(device=dev).manual_seed(4000 + li)
        copies = max(2, -(-3 * 129 * 2 ** 20 // (N * K)))
        qws = [torch.randint(-31, 32, (N, K), generator=g, device=dev, dtype=torch.int32).to(torch.int8)
               for _ in range(copies)]
        sw = torch.rand(N, generator=g, device=dev) * 1e-3
        bf = torch.zeros(N, device=dev)
        for M in (1, 16, 128, 1024, 4096):
            q = torch.randint(-31, 32, (M, K), generator=g, device=dev, dtype=torch.int32).half()
            y = torch.empty(M, N, dtype=torch.float16, device=dev)
            n = reps if M <= 128 else 4

            def calls():
                for i in range(n):
                    binding.ot_linear(q, qws[i % copies], sw, bf, 6, 6, y, workspace=ws)
            ms = _graph_ms(calls, n)
            ms16 = _fp16_gemm_ms(dev, M, N, K, n)
            ops = 2 * M * N * K
            t_roof = max(N * K / (peaks["hbm"] * 1e9), ops / (peaks["bf16"] * 1e12))
            pt = {"layer": layer.name, "K": K, "N": N, "tokens": M, "us": round(ms * 1e3, 2),
                  "tops": round(ops / (ms * 1e-3) / 1e12, 1),
                  "weight_gbs": round(N * K / (ms * 1e-3) / 1e9, 1),
                  "bound": "hbm" if N * K / (peaks["hbm"] * 1e9) > ops / (peaks["bf16"] * 1e12) else "tensor",
                  "frac_roofline": round(t_roof / (ms * 1e-3), 4),
                  "cublas_fp16_us": round(ms16 * 1e3, 2), "speedup_vs_fp16": round(ms16 / ms, 3)}
            if M <= 128:
                # int8 codes in, and the quantization inside the linear (fp16 X in), against
                # the quantize kernel followed by the linear
                q8 = q.to(torch.int8)
                x = q.clone()
                z0, r1 = torch.zeros(K, device=dev), torch.ones(K, device=dev)
                qs = torch.empty_like(q)

                def calls8():
                    for i in range(n):
                        binding.ot_linear(q8, qws[i % copies], sw, bf, 6, 6, y, workspace=ws)

                def calls_fused():
                    for i in range(n):
                        binding.ot_linear_fused(x, z0, r1, 6, qws[i % copies], sw, bf, 6, qs, y, workspace=ws)

                def calls_producer():
                    for i in range(n):
                        binding.ot_linear_fused(x, z0, r1, 6, qws[i % copies], sw, bf, 6, qs, y, workspace=ws,
                                                mode=binding.OT_FUSE_PRODUCER)

                def calls_two():
                    for i in range(n):
                        binding.ot_quantize_act(x, z0, r1, 6, qs, binding.OT_CODE_F16)
                        binding.ot_linear(qs, qws[i % copies], sw, bf, 6, 6, y, workspace=ws)
                pt["int8_codes_us"] = round(_graph_ms(calls8, n) * 1e3, 2)
                pt["fused_us"] = round(_graph_ms(calls_fused, n) * 1e3, 2)
                pt["fused_in_producer_us"] = round(_graph_ms(calls_producer, n) * 1e3, 2)
                pt["quantize_then_linear_us"] = round(_graph_ms(calls_two, n) * 1e3, 2)
                del q8, x, qs
            out.append(pt)
            del q, y
        del qws
    del ws
    torch.cuda.empty_cache()
    return {"workload": "opt-13b QKV and fc2, Int6, 1-4096 tokens", "timing": "CUDA graph replay, rotating weights",
            "up_to_128_tokens": "int8_codes_us: ot_linear on int8 codes; fused_us: ot_linear_fused (default: the "
                                "quantize kernel, the linear its programmatic dependent); fused_in_producer_us: "
                                "ot_linear_fused with the quantization in the linear's token producer; "
                                "quantize_then_linear_us: ot_quantize_act + ot_linear",
            "per_point": out}


def _fp16_gemm_ms(dev, M, N, K, reps):
    """cuBLAS fp16 (torch.matmul) of [M, K] x [K, N] with fp16 weights W [N, K],
    timed like the quantized linear beside it: `reps` consecutive calls that
    rotate over enough weight copies to exceed 3x the L2, replayed from a CUDA
    graph; ms per call."""
    import torch
    g = torch.Generator(device=dev).manual_seed(5000 + M)
    copies = max(2, -(-3 * L2_BYTES // (2 * N * K)))
    ws = [(torch.randn(N, K, generator=g, device=dev) * 0.02).half() for _ in range(copies)]
    x = torch.randn(M, K, generator=g, device=dev).half()
    y = torch.empty(M, N, dtype=torch.float16, device=dev)

    def calls():
        for i in range(reps):
            torch.matmul(x, ws[i % copies].t(), out=y)
    ms = _graph_ms(calls, reps)
    del ws, x, y
    return ms


def bench_quantize_sweep(dev, peaks, reps: int = 20):
    """The quantize kernel alone on OPT-6.7B-wide activations (K = 4096) from
    2048 to 65,536 tokens (34 MB to 1.07 GB of traffic), L2 flushed before each
    launch: small launches are bound by launch and first-load latency like a
    plain copy, large ones by HBM bandwidth."""
    import torch

    from paper_2406_18832_gb300 import binding
    K = 4096
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    g = torch.Generator(device=dev).manual_seed(77)
    z = torch.randn(K, generator=g, device=dev)
    r = torch.rand(K, generator=g, device=dev) * 10 + 1
    out = []
    for M in (2048, 8192, 65536):
        x = (torch.randn(M, K, generator=g, device=dev) * 4).half()
        q = torch.empty(M, K, dtype=torch.float16, device=dev)
        y = torch.empty_like(x)

        def med(fn):
            for _ in range(3):
                fn()
            ts = []
            for _ in range(reps):
                flush.fill_(1)
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                fn()
                e1.record()
                torch.cuda.synchronize()
                ts.append(e0.elapsed_time(e1))
            return statistics.median(ts)
        ms = med(lambda: binding.ot_quantize_act(x, z, r, 8, q, binding.OT_CODE_F16))
        mc = med(lambda: y.copy_(x))
        byt = 4 * M * K + 8 * K
        out.append({"tokens": M, "bytes": byt, "us": round(ms * 1e3, 2), "gbs": round(byt / (ms * 1e-3) / 1e9, 1),
                    "frac_hbm": round(byt / (ms * 1e-3) / 1e9 / peaks["hbm"], 4),
                    "torch_copy_gbs": round(4 * M * K / (mc * 1e-3) / 1e9, 1)})
        del x, q, y
    del flush
    torch.cuda.empty_cache()
    return {"workload": "quantize_kernel, K = 4096, fp16 X in + fp16 codes out", "l2": "flushed before each launch",
            "per_size": out}


def bench_layernorm(dev, peaks, reps: int = 200):
    """The LayerNorm before QKV / fc1 fused with the symmetrization and the
    per-channel quantization (Section 3.2), OPT-6.7B at 2048 tokens (hidden
    4096): one kernel reads h and writes the codes, against the unfused pair
    (a LayerNorm writing fp16, here torch's, then the quantize kernel).
    Consecutive calls rotate over input copies larger than the L2 and are
    timed as CUDA-graph replays."""
    import torch
    import torch.nn.functional as F

    from paper_2406_18832_gb300 import binding
    M, K, eps = STEP6_TOKENS, 4096, 1e-5
    g = torch.Generator(device=dev).manual_seed(77)
    copies = -(-3 * L2_BYTES // (M * K * 2))
    hs = [torch.randn(M, K, generator=g, device=dev).half() for _ in range(copies)]
    gamma = (1 + 0.1 * torch.randn(K, generator=g, device=dev)).half()
    beta = (0.1 * torch.randn(K, generator=g, device=dev)).half()
    z = 0.1 * torch.randn(K, generator=g, device=dev)
    r = torch.full((K,), 30.0, device=dev)
    gr, br = torch.empty(K, device=dev), torch.empty(K, device=dev)
    binding.ot_fold_layernorm(gamma, beta, z, r, gr, br)
    q = torch.empty(M, K, dtype=torch.float16, device=dev)

    def timed(fn):
        # CUDA-graph replay of `reps` consecutive calls (kernel time, not the
        # Python call overhead of eager launches)
        for i in range(copies):
            fn(hs[i])
        torch.cuda.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            for i in range(reps):
                fn(hs[i % copies])
        graph.replay()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(3):
            graph.replay()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / (3 * reps)

    fused_ms = timed(lambda h: binding.ot_layernorm_quantize(h, gr, br, eps, 8, q))

    def unfused(h):
        binding.ot_quantize_act(F.layer_norm(h, (K,), gamma, beta, eps), z, r, 8, q)

    unfused_ms = timed(unfused)
    bytes_fused = 4 * M * K + 8 * K
    gbs = bytes_fused / (fused_ms * 1e-3) / 1e9
    return {"workload": "opt-6.7b LayerNorm -> QKV / fc1 input, 2048 tokens x 4096", "kernel": "layernorm_quantize",
            "us": round(fused_ms * 1e3, 2), "gbs": round(gbs, 1), "frac_hbm": round(gbs / peaks["hbm"], 4),
            "bytes": bytes_fused, "note": "fp16 h in + fp16 codes out; statistics exact (integer sums)",
            "unfused_us": round(unfused_ms * 1e3, 2),
            "unfused": "torch layer_norm (fp16 out) + quantize_kernel"}


def bench_clipping(dev, peaks, minmax, reps: int = 3):
    """Token-wise clipping calibration (Appendix D) on the OPT-6.7B QKV
    calibration set (65,536 tokens x 4096, 512 MiB): per-channel order
    statistics by a two-pass radix select, against the one-pass min / max
    calibration of the same set (minmax = (ms, config) from the OPT-6.7B step)."""
    import torch

    from paper_2406_18832_gb300 import binding, synth
    minmax_ms, cfg_index = minmax
    cfg = synth.CONFIGS[cfg_index]
    layer = cfg.layers[0]
    x = synth.activations(cfg_index, 0, layer, cfg.T_cal, 3, device=dev)
    lo = torch.empty(layer.K, device=dev)
    hi = torch.empty(layer.K, device=dev)
    binding.ot_calibrate_clipped(x, 0.999, lo, hi)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        binding.ot_calibrate_clipped(x, 0.999, lo, hi)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    nbytes = x.numel() * 2
    del x
    return {"workload": "opt-6.7b QKV calibration set, 65536 tokens x 4096, alpha 0.999", "ms": round(ms, 3),
            "data_gbs": round(nbytes / (ms * 1e-3) / 1e9, 1),
            "read_gbs": round(2 * nbytes / (ms * 1e-3) / 1e9, 1),
            "frac_hbm": round(2 * nbytes / (ms * 1e-3) / 1e9 / peaks["hbm"], 4),
            "minmax_ms": round(minmax_ms, 3), "note": "two passes over the data (radix select on fp16 keys)"}


def _warm_graph(graph, min_s: float = 0.05):
    """Replay `graph` until at least `min_s` seconds of it have run (three
    replays at least).  A point that follows a long high-power one (the block,
    the headline step, the 4096-token points of the sweep) otherwise times
    while the clocks are still recovering: measured, such a decode point ran
    15-25 % slow in some runs."""
    import torch
    t0 = time.perf_counter()
    n = 0
    while n < 3 or time.perf_counter() - t0 < min_s:
        graph.replay()
        torch.cuda.synchronize()
        n += 1


def _graph_ms(calls, reps):
    """ms per call of `calls` (reps calls) captured in a CUDA graph: warm-up
    replays (_warm_graph), then the median of three timed rounds of five
    replays."""
    import torch
    calls()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        calls()
    _warm_graph(graph)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    rounds = []
    for _ in range(3):
        e0.record()
        for _ in range(5):
            graph.replay()
        e1.record()
        torch.cuda.synchronize()
        rounds.append(e0.elapsed_time(e1) / (5 * reps))
    del graph
    return statistics.median(rounds)


def bench_decode(dev, peaks, reps: int = 50):
    """Decode-sized linears of the OPT-13B shapes (Int6; 1 and 16 tokens): the
    product is bound by streaming the int8 weights from HBM, so the roofline is
    weight bytes / time against the HBM peak.  Decode steps are served as CUDA
    graphs, so the headline time per call is a replay of `reps` captured calls;
    the eager time (one C-ABI call from Python each) is reported beside it."""
    import torch

    from paper_2406_18832_gb300 import binding, synth
    c = synth.CONFIGS[3]
    res = []
    ws = torch.zeros(binding.ot_linear_workspace_size(), dtype=torch.uint8, device=dev)
    for li in (0, 3):
        layer = c.layers[li]
        qm = 31
        g = torch.Generator(device=dev).manual_seed(3000 + li)
        # as many weight copies (successive layers of the model) as keep the
        # weights read by consecutive calls above 3x the 129 MB L2
        copies = max(2, -(-3 * 129 * 2 ** 20 // (layer.N * layer.K)))
        qws = [torch.randint(-qm, qm + 1, (layer.N, layer.K), generator=g, device=dev,
                             dtype=torch.int32).to(torch.int8) for _ in range(copies)]
        sw = torch.rand(layer.N, generator=g, device=dev) * 1e-3
        bf = torch.zeros(layer.N, device=dev)
        for M in (1, 16):
            q = torch.randint(-qm, qm + 1, (M, layer.K), generator=g, device=dev, dtype=torch.int32).half()
            y = torch.empty(M, layer.N, dtype=torch.float16, device=dev)

            def calls():
                for i in range(reps):
                    binding.ot_linear(q, qws[i % copies], sw, bf, 6, 6, y, workspace=ws)

            ms = _graph_ms(calls, reps)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            calls()
            e1.record()
            torch.cuda.synchronize()
            eager_ms = e0.elapsed_time(e1) / reps
            gbs = layer.N * layer.K / (ms * 1e-3) / 1e9
            # with the activation quantization in front: two calls, or the
            # fused call (the linear a programmatic dependent of the quantize)
            x = q.clone()
            z0, r1 = torch.zeros(layer.K, device=dev), torch.ones(layer.K, device=dev)
            qs = torch.empty_like(q)

            def two_calls():
                for i in range(reps):
                    binding.ot_quantize_act(x, z0, r1, 6, qs, binding.OT_CODE_F16)
                    binding.ot_linear(qs, qws[i % copies], sw, bf, 6, 6, y, workspace=ws)

            def fused_calls():
                for i in range(reps):
                    binding.ot_linear_fused(x, z0, r1, 6, qws[i % copies], sw, bf, 6, qs, y, workspace=ws)

            ms_two, ms_fused = _graph_ms(two_calls, reps), _graph_ms(fused_calls, reps)
            ms16 = _fp16_gemm_ms(dev, M, layer.N, layer.K, reps)
            res.append({"layer": layer.name, "K": layer.K, "N": layer.N, "tokens": M, "us": round(ms * 1e3, 2),
                        "weight_gbs": round(gbs, 1), "frac_hbm": round(gbs / peaks["hbm"], 4),
                        "eager_us": round(eager_ms * 1e3, 2), "quantize_then_linear_us": round(ms_two * 1e3, 2),
                        "fused_us": round(ms_fused * 1e3, 2), "cublas_fp16_us": round(ms16 * 1e3, 2),
                        "speedup_vs_fp16": round(ms16 / ms, 3), "fused_speedup_vs_fp16": round(ms16 / ms_fused, 3)})
        del qws
    return {"workload": "opt-13b decode-sized linears, Int6", "kernel": "linear_gemv_kernel (mma.sync, TMA stream)",
            "bound": "hbm", "timing": "CUDA graph replay of consecutive calls (eager_us: one Python call each); "
            "quantize_then_linear_us / fused_us: ot_quantize_act + ot_linear per call, or ot_linear_fused; "
            "cublas_fp16_us: torch.matmul fp16 of the same shape, fp16 weights, timed the same way",
            "l2": "consecutive calls read different weight copies, > 3x L2 in all",
            "per_shape": res}


def bench_block(dev, tokens: int = 4096, t_cal: int = 4096, reps: int = 20):
    """The chained linear path of an OPT-30B-shaped decoder block (hidden 7168,
    FFN 28672; QKV -> V slice -> out -> fc1 + ReLU -> fc2, each layer calibrated
    on what it receives) at 8 x 512 tokens, Int8 and Int6: latency, weight and
    activation bytes against the same chain of cuBLAS fp16 GEMMs; also with
    fc1's epilogue writing fc2's codes (the chained epilogue)."""
    import torch

    from paper_2406_18832_gb300 import QuantizedBlockLinears, synth
    c = synth.CONFIGS[5]
    h, ffn = 7168, 28672
    weights = [synth.weights(5, i, layer, device=dev) for i, layer in enumerate(c.layers)]
    x_cal = synth.activations(5, 0, c.layers[0], t_cal, 3, device=dev)
    x = synth.activations(5, 0, c.layers[0], tokens, 4, device=dev)
    ops = 2 * tokens * sum(l.K * l.N for l in c.layers)

    def timed(fn):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            fn()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / reps

    out = {"workload": "opt-30b-block-linears", "tokens": tokens, "calibration_tokens": t_cal,
           "ops": ops, "reps": reps}
    for bits in (8, 6):
        blk = QuantizedBlockLinears(h, ffn, bits, bits, device=dev)
        blk.calibrate(x_cal, weights)
        ms = timed(lambda: blk.forward(x))
        # fc1's epilogue writes fc2's codes: f is neither written nor re-read
        ms_f = timed(lambda: blk.forward(x, fused=True))
        out[f"int{bits}"] = {"ms": round(ms, 4), "tops": round(ops / (ms * 1e-3) / 1e12, 1),
                             "ms_fc1_fc2_chained": round(ms_f, 4),
                             "tops_fc1_fc2_chained": round(ops / (ms_f * 1e-3) / 1e12, 1),
                             "weight_bytes": blk.weight_bytes()}
        del blk
    w16 = [w for w, _ in weights]
    b16 = [b for _, b in weights]

    def fp16_chain():
        qkv = torch.addmm(b16[0], x, w16[0].t())
        o = torch.addmm(b16[1], qkv[:, 2 * h:], w16[1].t())
        f = torch.relu(torch.addmm(b16[2], o, w16[2].t()))
        return torch.addmm(b16[3], f, w16[3].t())
    ms16 = timed(fp16_chain)
    out["cublas_fp16"] = {"ms": round(ms16, 4), "tflops": round(ops / (ms16 * 1e-3) / 1e12, 1),
                          "weight_bytes": sum(w.numel() * 2 + b.numel() * 2 for w, b in weights)}
    # activation bytes per block: fp16 inputs read (x, v, o, f) and outputs written
    # (qkv, o, f, y); the quantized path also writes and reads each layer's fp16 codes
    act16 = 2 * tokens * ((h + h + h + ffn) + (3 * h + h + ffn + h))
    quant = act16 + 4 * tokens * (h + h + h + ffn)
    out["activation_bytes"] = {"fp16_path": act16, "quantized_path": quant,
                               "quantized_fc1_fc2_chained": quant - 4 * tokens * ffn}
    del weights, x_cal, x
    torch.cuda.empty_cache()
    return out


def bench_per_token(dev, peaks, reps: int = 50):
    """The per-token path (Eq. 3) the paper uses for the out and fc2 linears:
    dynamic per-token scales and codes (one kernel), then the linear with the
    per-token x per-channel epilogue, OPT-6.7B out (4096 -> 4096) and fc2
    (16384 -> 4096) at 2048 tokens, W8A8, against the per-channel step of
    the same shapes (static z, r) and cuBLAS fp16.  Consecutive calls replayed
    from a CUDA graph."""
    import torch

    from paper_2406_18832_gb300 import binding, synth
    c = synth.CONFIGS[STEP6_CFG]
    M = STEP6_TOKENS
    ws = torch.zeros(binding.ot_linear_workspace_size(), dtype=torch.uint8, device=dev)
    out = []
    for li in (1, 3):
        layer = c.layers[li]
        K, N = layer.K, layer.N
        w, b = synth.weights(STEP6_CFG, li, layer, device=dev)
        x = synth.activations(STEP6_CFG, li, layer, M, 4, device=dev)
        qw = torch.empty(N, K, dtype=torch.int8, device=dev)
        sw = torch.empty(N, device=dev)
        binding.ot_quantize_weights(w, 8, qw, sw)
        bias = b.float()
        q = torch.empty(M, K, dtype=torch.float16, device=dev)
        s_tok = torch.empty(M, device=dev)
        y = torch.empty(M, N, dtype=torch.float16, device=dev)

        def tok_calls():
            for _ in range(reps):
                binding.ot_quantize_tokens(x, 8, q, s_tok)
                binding.ot_linear_per_token(q, qw, sw, s_tok, bias, 8, 8, y, workspace=ws)

        def quant_only():
            for _ in range(reps):
                binding.ot_quantize_tokens(x, 8, q, s_tok)
        ms = _graph_ms(tok_calls, reps)
        ms_q = _graph_ms(quant_only, reps)
        ops = 2 * M * N * K
        out.append({"layer": layer.name, "K": K, "N": N, "tokens": M, "us": round(ms * 1e3, 2),
                    "tops": round(ops / (ms * 1e-3) / 1e12, 1), "quantize_tokens_us": round(ms_q * 1e3, 2),
                    "quantize_tokens_gbs": round((3 * M * K + 4 * M) / (ms_q * 1e-3) / 1e9, 1)})
        del w, b, x, qw, q, y
    del ws
    torch.cuda.empty_cache()
    return {"workload": "opt-6.7b out and fc2 at 2048 tokens, per-token activations (Eq. 3), W8A8",
            "timing": "CUDA graph replay; quantize_tokens reads each row twice (max, then codes; the second "
                      "read mostly from L2); gbs on fp16 X in + int8 codes out + scales",
            "per_layer": out}


# ----------------------------------------------------------------------------
# the CPU oracle (baseline leg and --impl reference)
# ----------------------------------------------------------------------------
def _oracle_fold_layers(host, bits, timings):
    """Calibrate (on each layer's calibration sample), derive the parameters
    and fold the whole layer with the oracle, timing each step."""
    import oracle
    out = []
    for d in host:
        t = time.perf_counter()
        mn, mx = oracle.calibrate_mt(d["xc"])
        timings["calibrate_s"] += time.perf_counter() - t
        timings["calibrate_bytes"] += d["xc"].nbytes
        t = time.perf_counter()
        z, s, r = oracle.params(mn, mx, bits[0])
        timings["params_s"] += time.perf_counter() - t
        t = time.perf_counter()
        qw, sw, bf = oracle.fold_mt(d["w"], d["b"], z, s, bits[1])
        timings["fold_s"] += time.perf_counter() - t
        timings["fold_weights"] += d["w"].size
        out.append(dict(z=z, r=r, qw=qw, sw=sw, bf=bf, relu=d["relu"], K=d["w"].shape[1], N=d["w"].shape[0]))
    return out


def _oracle_tokens(ol, xs, rows, bits, timings):
    """The online steps (quantize, int64 product, fp32-fma epilogue) of `rows`
    tokens through every layer with the oracle's threaded drivers; returns ops."""
    import oracle
    ops = 0
    for d, x in zip(ol, xs):
        xr = x[rows]
        t = time.perf_counter()
        q = oracle.quantize_mt(xr, d["z"], d["r"], bits[0])
        t1 = time.perf_counter()
        acc = oracle.matmul_mt(q, d["qw"])
        t2 = time.perf_counter()
        oracle.epilogue_mt(acc, d["sw"], d["bf"], d["relu"])
        t3 = time.perf_counter()
        timings["quantize_s"] += t1 - t
        timings["matmul_s"] += t2 - t1
        timings["epilogue_s"] += t3 - t2
        ops += 2 * len(rows) * d["N"] * d["K"]
    return ops


def _new_timings():
    return dict(calibrate_s=0.0, calibrate_bytes=0, params_s=0.0, fold_s=0.0, fold_weights=0,
                quantize_s=0.0, matmul_s=0.0, epilogue_s=0.0)


def cpu_single_thread():
    """The oracle's plain C functions on one host thread: config 1's whole step
    (calibration on its 64 tokens, parameters, fold, then quantize / int64
    product / epilogue of its 16 tokens) and config 2's out layer (4096 ->
    4096; calibration on 2048 tokens, the whole fold, a 64-token sample of the
    online steps).  Seconds per step and online TOPS."""
    import numpy as np

    import oracle
    from paper_2406_18832_gb300 import synth
    out = {}
    for name, cfg, li, tokens, cal in (("config1", 1, 0, 16, 64), ("config2_out", 2, 1, 64, 2048)):
        layer = synth.CONFIGS[cfg].layers[li]
        w, b = synth.weights(cfg, li, layer)
        xc = synth.activations(cfg, li, layer, cal, 3).numpy()
        x = synth.activations(cfg, li, layer, tokens, 4).numpy()
        w, b = w.numpy(), b.numpy()
        st = {}
        t = time.perf_counter()
        mn, mx = oracle.calibrate(xc)
        st["calibrate"] = time.perf_counter() - t
        t = time.perf_counter()
        z, s_, r = oracle.params(mn, mx, 8)
        st["params"] = time.perf_counter() - t
        t = time.perf_counter()
        qw, sw, bf = oracle.fold(w, b, z, s_, 8)
        st["fold"] = time.perf_counter() - t
        t = time.perf_counter()
        q = oracle.quantize(x, z, r, 8)
        st["quantize"] = time.perf_counter() - t
        t = time.perf_counter()
        acc = oracle.matmul(q, qw)
        st["matmul"] = time.perf_counter() - t
        t = time.perf_counter()
        oracle.epilogue(acc, sw, bf, layer.relu_out)
        st["epilogue"] = time.perf_counter() - t
        online = st["quantize"] + st["matmul"] + st["epilogue"]
        out[name] = {"tokens": tokens, "K": layer.K, "N": layer.N, "calibration_tokens": cal,
                     "per_step_s": {k: round(v, 6) for k, v in st.items()},
                     "online_tops": round(2.0 * tokens * layer.K * layer.N / online / 1e12, 6)}
    return out


def cpu_baseline(host, budget_s=12.0):
    """Time the oracle, as it stands, per step of the headline workload on the
    host cores (its C functions over row ranges in one thread per core):
    calibration on 8192 tokens per layer, parameters, the fold of the whole
    layers, then quantize / int64 product / epilogue of a token sample sized
    to about `budget_s` seconds.  value = online ops / online seconds."""
    import numpy as np

    import oracle
    tm = _new_timings()
    ol = _oracle_fold_layers(host, BITS, tm)
    xs = [d["x"] for d in host]
    probe = _new_timings()
    t = time.perf_counter()
    _oracle_tokens(ol, xs, np.arange(16), BITS, probe)
    per16 = time.perf_counter() - t
    rows_n = int(max(16, min(xs[0].shape[0], budget_s / max(per16, 1e-6) * 16)) // 16 * 16)
    ops = _oracle_tokens(ol, xs, np.arange(rows_n), BITS, tm)
    online = tm["quantize_s"] + tm["matmul_s"] + tm["epilogue_s"]
    cores = oracle.host_threads()
    return {"value": round(ops / online / 1e12, 6), "unit": "TOPS", "cores": cores, "kind": "oracle",
            "sample": f"{rows_n} of the {TOKENS} tokens through fc1 and fc2 (quantize, int64 product, fp32-fma "
                      f"epilogue, {online:.1f} s); offline steps: calibration on 8192 tokens per layer, "
                      f"parameters, the fold of both whole layers",
            "per_step_s": {"calibrate": round(tm["calibrate_s"], 3), "params": round(tm["params_s"], 5),
                           "fold": round(tm["fold_s"], 3), "quantize": round(tm["quantize_s"], 3),
                           "matmul": round(tm["matmul_s"], 3), "epilogue": round(tm["epilogue_s"], 3)},
            "calibrate_gbs": round(tm["calibrate_bytes"] / tm["calibrate_s"] / 1e9, 2),
            "fold_mweights_per_s": round(tm["fold_weights"] / tm["fold_s"] / 1e6, 1),
            "threads": "one per core of os.sched_getaffinity, rows (or channels) split evenly",
            "single_thread": cpu_single_thread()}


def run_reference(args):
    """The CPU oracle on the headline workload (inputs drawn on the host), one
    step = a bounded token sample through fc1 and fc2, sized so warm-up and
    timed steps end within about two minutes."""
    import numpy as np

    import oracle
    from paper_2406_18832_gb300 import synth
    rank, world, _ = _env_rank()
    if rank != 0:
        return
    cfg, layer_shapes = _workload_desc()
    host = []
    for li, layer in enumerate(cfg.layers):
        w, b = synth.weights(WORKLOAD_CFG, li, layer)
        host.append(dict(w=w.numpy(), b=b.numpy(), relu=layer.relu_out,
                         xc=synth.activations(WORKLOAD_CFG, li, layer, 2048, 3).numpy(),
                         x=synth.activations(WORKLOAD_CFG, li, layer, TOKENS, 4).numpy()))
    setup = _new_timings()
    ol = _oracle_fold_layers(host, BITS, setup)
    xs = [d["x"] for d in host]
    probe = _new_timings()
    t = time.perf_counter()
    _oracle_tokens(ol, xs, np.arange(8), BITS, probe)
    per8 = time.perf_counter() - t
    budget_step = max(0.05, 110.0 / max(1, args.steps + args.warmup))
    rows_n = int(max(1, min(TOKENS, budget_step / max(per8, 1e-6) * 8)))
    for k in range(args.warmup):
        _oracle_tokens(ol, xs, (np.arange(rows_n) + k * rows_n) % TOKENS, BITS, _new_timings())
    tm = _new_timings()
    t = time.perf_counter()
    ops = 0
    for k in range(args.steps):
        ops += _oracle_tokens(ol, xs, (np.arange(rows_n) + (k + args.warmup) * rows_n) % TOKENS, BITS, tm)
    dt = time.perf_counter() - t
    value = ops / dt / 1e12
    cores = oracle.host_threads()
    sample = (f"per step: {rows_n} of the {TOKENS} tokens through fc1 and fc2 (quantize, int64 product, "
              f"fp32-fma epilogue) on {cores} host threads; weights folded once before timing")
    line = {"metric": METRIC, "value": round(value, 6), "unit": "TOPS", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(dt / args.steps * 1e3, 4), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "int64 (CPU oracle)", "data": "synthetic",
            "impl": "reference",
            "config": {"workload": WORKLOAD_NAME, "tokens": TOKENS, "bits_a": BITS[0], "bits_w": BITS[1],
                       "layers": [{"name": n, "K": K, "N": N} for n, K, N in layer_shapes]},
            "cpu_baseline": {"value": round(value, 6), "unit": "TOPS", "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": round(value, 6), "unit": "TOPS", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--cpu-budget", type=float, default=12.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-block", action="store_true", help="skip the OPT-30B block stage")
    ap.add_argument("--profile-decode", action="store_true",
                    help="profiler run of the decode-sized linears only (after the setup)")
    ap.add_argument("--profile", action="store_true",
                    help="profiler run: 8192 calibration tokens, the timed steps only, no report")
    ap.add_argument("--profile-opt67b", action="store_true",
                    help="for profilers: only the OPT-6.7B step (2048 tokens), warmup + steps times")
    ap.add_argument("--profile-linear", type=int, default=0, metavar="TOKENS",
                    help="profiler run of the OPT-13B QKV and fc2 linears at TOKENS tokens only")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
