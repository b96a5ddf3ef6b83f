#!/usr/bin/env python
"""ZO-step throughput of the ZO-Act hot path on GB300.

Default workload: the full Llama-3-8B linear stack in bf16 -- 32 decoder layers
x {q 4096->4096, k/v 4096->1024, o 4096->4096, gate/up 4096->14336, down
14336->4096} = 224 adapted linears, r = 16, T = 16 x 256 = 4096 tokens per
perturbation (8192 stacked rows for the +/- pair), each layer's input the
RMS-normalised output before it, loss = mean squared output, eps = 1e-3, Adam
on all 22.0 M coefficients.  Other workloads (--workload): llama_mlp_bf16 (the
MLP block: gate/up 4096 -> 14336 on a shared input, down 14336 -> 4096, MSE to
N(0,1) targets, T = 2048), llama_stack_int4 (the stack with INT4 g128 weights),
opt_stack_fp16 (240 linears, r = 32).  Synthetic data: rank-64 Gaussian signal
plus 5% noise, unit RMS per token; W ~ N(0, 0.02).  The bases come from
Algorithm 1 on the device before timing: one calibration forward pass of the
base model, then zoact_basis_init on every layer's input.

One step = per adapted linear zoact_lowrank_proj + zoact_pair_forward (gate/up:
zoact_pair_forward_gated) with the glue ops, then zoact_loss_pair and
zoact_adam_step, all on one stream, no host synchronisation.

value = training tokens/s = world_size * T / step time (CUDA events around
exactly --steps steps, max over ranks).  The frozen weights are larger than L2
(129 MB), so every step reads them from HBM.  `--impl reference` times the CPU
oracle (numpy fp64) on a bounded sample of the default workload instead.
`--measure-peak fp16` measures the dense fp16 tensor peak the OPT-13B workload
is graded against; `--measure-read` times the loss launch (and torch.sum) on
50 MB to 805 MB reads.
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "ZO-step tokens/s per adapted-linear stack; % of HBM or tensor-pipe roofline"
UNIT = "tokens/s"
DEFAULT_WORKLOAD = "llama_stack_bf16"
N_CAL = {"llama_mlp_bf16": 2048, "llama_stack_bf16": 512, "llama_stack_int4": 512, "opt_stack_fp16": 4096}
LR = 1e-4
TIMING_PAIRS = 4096          # event pairs in the library's kernel-timing pool (launches timed per read)


# DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum) of one step's pair launches, from ncu captures of
# the current kernels; workloads without such a capture report null.  The stacks' are scaled from 2-decoder
# captures (`--decoders 2`): decoder 0 plus (decoders - 1) times decoder 1 (the later decoders have its shapes);
# the INT4 stack's include the expansions of W timed with their pair launches.  A run with a kernel switch set
# (other kernels than the captured ones) reports null.
PAIR_TRAFFIC_BYTES = {"llama_stack_bf16": 82.95e9, "llama_mlp_bf16": 933.9e6, "opt_stack_fp16": 208.66e9,
                      "llama_stack_int4": 91.08e9}
KERNEL_SWITCHES = ("ZOACT_INT4", "ZOACT_PAIR_KERNEL", "ZOACT_LOWRANK", "ZOACT_GROUP_M", "ZOACT_SPLIT_TAIL")


# Dense fp16 tensor peak of the GB300s (TFLOP/s), measured like the bf16 peaks of MEASURED_PEAKS.json
# with `python bench.py --measure-peak fp16`: torch.matmul fp16 8192^3, best of 10 (burst) and back to back
# for 4 s (sustained, under the power cap).  The same command for bf16 gave 1924.6 / 1735.2 on that box
# (MEASURED_PEAKS.json: 1910.6 / 1699.8).
FP16_PEAKS = {"burst": 1819.3, "sustained": 1640.4}


def _peaks(dtype="bf16"):
    """(HBM GB/s, dense burst TFLOP/s, dense sustained TFLOP/s, provenance) for the compute dtype."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        hbm, burst, sust, kind = p["hbm_gbs"], p["bf16_tflops"], p["bf16_tflops_sustained"], "measured"
    except Exception:
        hbm, burst, sust, kind = 6800.0, 1900.0, 1700.0, "fallback"
    if dtype == "fp16":
        if FP16_PEAKS is not None:
            return hbm, FP16_PEAKS["burst"], FP16_PEAKS["sustained"], "measured fp16"
        return hbm, burst, sust, kind + " (bf16 peak: fp16 not measured)"
    return hbm, burst, sust, kind


def measure_peak(dtype, seconds=4.0):
    """Dense tensor peak of one GPU: torch.matmul of 8192^3 in dtype, best of 10 (burst), and back-to-back
    matmuls for `seconds` (sustained), CUDA events; clocks sampled meanwhile."""
    import torch
    dt = {"fp16": torch.float16, "bf16": torch.bfloat16}[dtype]
    n = 8192
    g = torch.Generator(device="cuda").manual_seed(0)
    a = torch.randn(n, n, device="cuda", dtype=dt, generator=g)
    b = torch.randn(n, n, device="cuda", dtype=dt, generator=g)
    c = torch.empty(n, n, device="cuda", dtype=dt)
    flop = 2.0 * n ** 3
    for _ in range(5):
        torch.matmul(a, b, out=c)
    torch.cuda.synchronize()
    sampler = ClockSampler(torch.cuda.current_device())
    sampler.start()
    best = float("inf")
    for _ in range(10):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(); torch.matmul(a, b, out=c); e1.record()
        torch.cuda.synchronize()
        best = min(best, e0.elapsed_time(e1))
    reps, t_end = 0, time.time() + seconds
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    while time.time() < t_end:
        for _ in range(20):
            torch.matmul(a, b, out=c)
        reps += 20
        torch.cuda.synchronize()
    e1.record()
    torch.cuda.synchronize()
    clocks = sampler.stop()
    print(json.dumps({"peak": f"{dtype} dense", "shape": [n, n, n], "burst_tflops": flop / (best * 1e-3) / 1e12,
                      "sustained_tflops": flop * reps / (e0.elapsed_time(e1) * 1e-3) / 1e12,
                      "sustained_s": e0.elapsed_time(e1) * 1e-3, "matmuls": reps, "clocks": clocks,
                      "gpu": torch.cuda.get_device_name(), "torch": torch.__version__}))


def measure_read():
    """What one launch reading a given number of bytes reaches on this GPU.  zoact_loss_pair on the MLP block's
    loss shape (y+, y- and t: 2 x 2048 x 4096 and 2048 x 4096 bf16, 50.3 MB) and on 2, 4 and 16 times as many
    tokens, the projection (zoact_lowrank_proj_prepared, r = 16, split-K sum included) of an X of the same bytes,
    and torch.sum over a bf16 buffer of the same bytes; best of 10 by CUDA events, each after writing a 512 MB
    buffer (larger than L2).  An empty launch between the same events gives the events' own overhead (host
    dispatch included)."""
    import torch
    import paper_2607_01125_gb300 as zo
    ctx = zo.Context(torch.cuda.current_device())
    n_col = 4096
    base = 3 * 2048 * n_col                      # bf16 elements of the MLP block's loss pair
    buf = torch.ones(16 * base, device="cuda", dtype=torch.bfloat16)
    flush = torch.empty(512 << 20, device="cuda", dtype=torch.uint8)
    tiny = torch.zeros(1, device="cuda")
    loss_out = torch.zeros(4, device="cuda", dtype=torch.float64)
    # the projection P = X U (r = 16, the prepared basis) over X of the same bytes: [6144 mult, 4096] bf16
    U = torch.randn(n_col, 16, device="cuda") / n_col ** 0.5
    utc = torch.empty(zo.zoact_basis_prepared_bytes(n_col, 16), dtype=torch.uint8, device="cuda")
    zo.zoact_basis_prepare(ctx, U, zo.DT_BF16, utc)
    P = torch.empty(16 * 6144, 16, device="cuda")
    out = []

    def best_us(fn):
        best = float("inf")
        for r in range(12):
            flush.fill_(r)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(); fn(); e1.record()
            torch.cuda.synchronize()
            if r >= 2:
                best = min(best, e0.elapsed_time(e1) * 1e3)
        return best

    for mult in (1, 2, 4, 16):
        n = mult * base
        T = mult * 2048
        Y = buf[:2 * T * n_col].view(2 * T, n_col)
        tgt = buf[2 * T * n_col:3 * T * n_col].view(T, n_col)
        us_loss = best_us(lambda: zo.zoact_loss_pair(ctx, Y, T, 1e-3, loss_out, target=tgt))
        X = buf[:n].view(n // n_col, n_col)
        Pm = P[:n // n_col]
        us_proj = best_us(lambda: zo.zoact_lowrank_proj_prepared(ctx, X, utc, 16, Pm))
        us_sum = best_us(lambda: torch.sum(buf[:n]))
        out.append({"mbytes": round(2 * n / 1e6, 1), "zoact_loss_pair_us": round(us_loss, 2),
                    "zoact_loss_pair_tb_per_s": round(2 * n / us_loss / 1e6, 2),
                    "zoact_lowrank_proj_us": round(us_proj, 2),
                    "zoact_lowrank_proj_tb_per_s": round(2 * n / us_proj / 1e6, 2), "torch_sum_us": round(us_sum, 2),
                    "torch_sum_tb_per_s": round(2 * n / us_sum / 1e6, 2)})
    print(json.dumps({"read": "one launch, L2 flushed, CUDA events", "sizes": out,
                      "empty_launch_us": round(best_us(lambda: tiny.add_(0.0)), 2),
                      "device_status": ctx.device_status(), "gpu": torch.cuda.get_device_name(),
                      "torch": torch.__version__}))
    ctx.close()


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 100 ms in a child process."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        # the raw samples; BENCH_CLOCKS_DIR moves them (the JSON line carries their summary)
        self.path = os.path.join(os.environ.get("BENCH_CLOCKS_DIR", os.path.join(ROOT, "bench_clocks")),
                                 f"clocks_gpu{index}.csv")

    def start(self):
        os.makedirs(os.path.dirname(self.path), exist_ok=True)
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 8:
                    continue
                try:
                    sm.append(float(parts[0]))
                    smax.append(float(parts[1]))
                except ValueError:
                    continue
                for nm, v in zip(names, parts[4:8]):
                    if v.lower() == "active":
                        reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


def dist_setup():
    import torch
    import torch.distributed as dist
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1 and not dist.is_initialized():
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device(f"cuda:{local}"))
    return world, rank, local


def build(ctx, dev, rank, name, tokens=None, n_queries=None, r=None, n_decoder=None):
    """Weights, bases (Algorithm 1 on the device) and the ZOStep of a workload.

    Returns (step, x, target, basis_seconds, workload).  Weights and calibration tokens, hence the bases,
    are the same on every rank; the training tokens (in the calibration set's signal subspace) and the
    targets are drawn per rank.
    """
    import torch
    import paper_2607_01125_gb300 as zo
    from paper_2607_01125_gb300.model import AdaptedLinear, ZOStep, coefficient_offsets, calibrate_bases
    from synth import workload, normal, lowrank_activations, quantize_int4_g128, tensor_seed
    over = {}
    if tokens is not None:
        over["T"] = tokens
    if r is not None:
        over["r"] = r
    if n_decoder is not None:
        over["n_decoder"] = n_decoder
    w = workload(name, **over)
    dt = {"bf16": torch.bfloat16, "fp16": torch.float16}[w.act_dtype]
    specs = w.linears()
    offs = coefficient_offsets(specs, w.r)
    lins = []
    for s, off in zip(specs, offs):
        U = torch.zeros(s.d_in, w.r, device=dev)
        if w.wtype == "int4_g128":
            Wf = normal((s.d_out, s.d_in), tensor_seed(w, "W", s.name), dev, std=w.weight_std)
            packed, scales = quantize_int4_g128(Wf)
            del Wf
            lins.append(AdaptedLinear(s.name, packed, U, s.layer_id, off, w.r, w_scales=scales,
                                      wtype=zo.DT_INT4_G128, d_in=s.d_in))
        else:
            W = normal((s.d_out, s.d_in), tensor_seed(w, "W", s.name), dev, std=w.weight_std, dtype=dt)
            lins.append(AdaptedLinear(s.name, W, U, s.layer_id, off, w.r))
    n_cal = N_CAL[name]
    x_cal, B = lowrank_activations(n_cal, w.d_model, 64, 0.05, tensor_seed(w, "x"), dev, dtype=dt)
    x, _ = lowrank_activations(w.T, w.d_model, 64, 0.05, tensor_seed(w, "x", rank), dev, dtype=dt, basis=B)
    target = normal((w.T, w.d_model), tensor_seed(w, "target", rank), dev, dtype=dt) if w.kind == "llama_mlp" else None
    # Algorithm 1: calibration forward pass of the base model, one basis per layer input
    step_cal = ZOStep(ctx, w.kind, lins, n_cal, w.act_dtype, eps=w.eps)
    torch.cuda.synchronize()
    t0 = time.time()
    calibrate_bases(ctx, step_cal, x_cal, w.r, oversample=16, n_iter=8, seed=tensor_seed(w, "basis"))
    torch.cuda.synchronize()
    basis_s = time.time() - t0
    del step_cal
    step = ZOStep(ctx, w.kind, lins, w.T, w.act_dtype, eps=w.eps, lr=LR, n_queries=n_queries)
    return step, x, target, basis_s, w


def time_diagnostics(ctx, step, dev, reps=20):
    """Section 5.3 diagnostics on the first layer's basis: gradient-energy capture of a synthetic bf16
    gradient shaped like that layer's weight ([d_in, d_out]) and the overlap of the basis with a rotated copy.
    HBM-bound on G; reported with its achieved GB/s."""
    import torch
    import paper_2607_01125_gb300 as zo
    from synth import normal
    lin = step.linears[0]
    G = normal((lin.d_in, lin.d_out), 99, dev, dtype=torch.bfloat16)
    U2 = torch.linalg.qr(lin.U + 0.1 * normal(tuple(lin.U.shape), 98, dev))[0].contiguous()
    out = torch.zeros(3, dtype=torch.float64, device=dev)
    res = {}
    for name, fn, nbytes in (("gradient_energy", lambda: zo.zoact_gradient_energy(ctx, lin.U, G, out),
                              G.numel() * G.element_size()),
                             ("subspace_overlap", lambda: zo.zoact_subspace_overlap(ctx, lin.U, U2, out),
                              2 * lin.U.numel() * 4)):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            fn()
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / reps
        res[name] = {"ms": ms, "GB/s": nbytes / (ms * 1e-3) / 1e9, "value": float(out[2]),
                     "shape": [lin.d_in, lin.d_out if name == "gradient_energy" else lin.r]}
    return res


def run_step(step, x, target, t, seed, world):
    step.forward_loss(x, target, seed, t)            # the pair forwards, then the loss pair
    if world > 1:
        from paper_2607_01125_gb300.dp import allreduce_loss
        allreduce_loss(step.loss_out, ctx=step.ctx)   # losses and a's are means over equal token counts
    step.update(t, seed, t)
    return step.loss_out


def run_ours(args):
    import torch
    import torch.distributed as dist
    world, rank, local = dist_setup()
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_01125_gb300 as zo
    dev = f"cuda:{local}"
    torch.cuda.set_device(local)
    ctx = zo.Context(local)
    step, x, target, basis_s, w = build(ctx, dev, rank, args.workload, args.tokens, args.queries, args.rank,
                                        args.decoders)
    seed = 1234

    def barrier():
        if world > 1:
            dist.barrier()

    t = 1
    for _ in range(args.warmup):
        run_step(step, x, target, t, seed, world); t += 1
    sampler = ClockSampler(local)
    sampler.start()
    torch.cuda.synchronize()
    soak_end = time.time() + args.soak       # untimed steps so the clocks reach their loaded state
    while time.time() < soak_end:
        run_step(step, x, target, t, seed, world); t += 1
        torch.cuda.synchronize()

    # ---- timed region: exactly args.steps steps, no per-kernel instrumentation ----
    n0 = ctx.launch_count()
    barrier(); torch.cuda.synchronize()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.nvtx.range_push("timed")          # profilers select the timed steps by this range
    start.record()
    for _ in range(args.steps):
        run_step(step, x, target, t, seed, world); t += 1
    end.record()
    torch.cuda.nvtx.range_pop()
    torch.cuda.synchronize(); barrier()
    launches = ctx.launch_count() - n0
    ms = start.elapsed_time(end) / args.steps

    # ---- kernel timing: the steps again (as many as the library's pool of event pairs covers whole), with
    # the library recording CUDA events on its stream around every tensor-core pair-forward kernel (the
    # events themselves lengthen a step by a few per cent, so the throughput above is taken without them) ----
    step.flops = []
    run_step(step, x, target, t, seed, world); t += 1          # one untimed step counts the launches per step
    per_step = max(1, len(step.flops))
    instr_steps = max(1, min(args.steps, TIMING_PAIRS // per_step))
    step.flops = []
    ctx.kernel_timing(True)
    barrier(); torch.cuda.synchronize()
    i_s, i_e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    i_s.record()
    for _ in range(instr_steps):
        run_step(step, x, target, t, seed, world); t += 1
    i_e.record()
    torch.cuda.synchronize(); barrier()
    instr_ms = i_s.elapsed_time(i_e) / instr_steps
    kern_ms, kern_launches = ctx.kernel_time()
    ctx.kernel_timing(False)
    if kern_launches != len(step.flops):
        raise RuntimeError(f"timed {kern_launches} pair launches of {len(step.flops)}: the timing is incomplete")
    gemm_flops = sum(step.flops)
    step.flops = None

    # ---- end to end through the public API with host buffers: every step's inputs are copied from pinned
    # host memory (overlapped with the previous step on a side stream) and its loss vector read back.  The
    # feeder's device buffers, side stream and events are made before the timed region ----
    from paper_2607_01125_gb300.model import HostFeeder
    x_h = x.cpu().pin_memory()
    t_h = target.cpu().pin_memory() if target is not None else None
    outs_h = [torch.empty(step.loss_out.numel(), dtype=torch.float64).pin_memory() for _ in range(args.steps)]
    batches = [(x_h, t_h) if t_h is not None else (x_h,) for _ in range(args.steps)]
    feeder = HostFeeder(batches[0])
    t_e2e = t

    def e2e_step(dev, i):
        return run_step(step, dev[0], dev[1] if len(dev) > 1 else None, t_e2e + i, seed, world)

    barrier(); torch.cuda.synchronize()
    e_s, e_e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e_s.record()
    feeder.run(batches, e2e_step, outs_h)
    e_e.record()
    t += args.steps
    torch.cuda.synchronize(); barrier()
    clocks = sampler.stop()
    e2e_ms = e_s.elapsed_time(e_e) / args.steps
    status = ctx.device_status()
    replicas = None
    if world > 1:                               # every rank must still hold the same coefficients and moments
        from paper_2607_01125_gb300.dp import check_replicas
        st, bad = check_replicas([step.C, step.m, step.v], ctx=ctx)
        replicas = {"status": st, "ranks_differing_from_rank0": bad}

    if world > 1:
        tt = torch.tensor([ms, e2e_ms], device=dev)
        dist.all_reduce(tt, op=dist.ReduceOp.MAX)
        ms, e2e_ms = float(tt[0]), float(tt[1])
    if rank != 0:
        return
    hbm, tf_burst, tf_sust, peak_kind = _peaks(w.act_dtype)
    # a step of about a millisecond times its kernels as bursts; the stacks' ~100 ms steps use the sustained peak
    long_step = ms > 20.0
    peak = tf_sust if long_step else tf_burst
    # the dominant kernel's own launches (the pair-forward calls also run their operand preparation)
    achieved = gemm_flops / (kern_ms * 1e-3) / 1e12
    T = w.T
    h2d = x.numel() * x.element_size() + (target.numel() * target.element_size() if target is not None else 0)
    line = {
        "metric": METRIC, "value": world * T / (ms * 1e-3), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "int4-bf16" if w.wtype == "int4_g128" else w.act_dtype,
        "data": "synthetic",
        "config": {"workload": w.name if args.decoders is None else f"{w.name} ({w.n_decoder} decoders)",
                   "tokens_per_perturbation": T, "stacked_rows": step.nb * T, "r": w.r,
                   "eps": w.eps, "adapted_linears": len(w.linears()),
                   "estimator": "two-sided, q=1" if args.queries is None else f"one-sided, q={args.queries}",
                   "l2": "inputs larger than L2 (frozen weights streamed from HBM every step)",
                   "parallelism": f"dp{world}" if world > 1 else "single"},
        "evaluated_tokens_per_s": world * step.nb * T / (ms * 1e-3),
        "zo_steps_per_s": 1e3 / ms,
        "pair_kernel_ms_per_step": kern_ms / instr_steps,
        "instrumented_ms_per_step": instr_ms,
        "pair_kernel_launches": kern_launches,
        "instrumented_steps": instr_steps,
        "basis_init_s": basis_s,
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak,
                     "peak_kind": f"{w.act_dtype} dense {'sustained' if long_step else 'burst'}, {peak_kind}",
                     "kernel": "pair_tc2_kernel / pair_tc_kernel (every pair-forward launch of the step, "
                               "timed alone by events on the library's stream over a second run of the same "
                               "number of steps)",
                     "algorithmic_flops_per_step": gemm_flops / instr_steps,
                     "traffic": (PAIR_TRAFFIC_BYTES.get(w.name)
                                 if args.tokens is None and args.queries is None and args.rank is None
                                 and args.decoders is None and not any(os.environ.get(k) for k in KERNEL_SWITCHES)
                                 else None),
                     "traffic_unit": "bytes per step (all pair launches of the step)"},
        "e2e": {"value": world * T / (e2e_ms * 1e-3), "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": 8 * step.loss_out.numel()},
        "gpu_launches": launches,
        "clocks": clocks,
        "device_status": status,
    }
    if replicas is not None:
        line["replicas"] = replicas
    if args.diag:
        line["diag"] = time_diagnostics(ctx, step, dev)
    if world == 1 and not args.no_cpu_baseline and args.queries is None and args.rank is None:
        line["cpu_baseline"] = cpu_baseline(step, w, budget_s=args.cpu_budget)
    print(json.dumps(line))


def _oracle_step(lay, x, tgt, seed, query, t):
    import numpy as np
    from oracle import graphs, loss as oloss, optim, philox
    Y = graphs.llama_mlp_forward(lay, x, 1e-3, seed, query, store="bf16")
    _, _, _, a = oloss.loss_pair(Y, x.shape[0], tgt, 1e-3)
    for l in lay:
        gz = optim.zo_gradient(a, philox.perturbation(seed, l["layer_id"], query, *l["C"].shape))
        l.setdefault("m", np.zeros_like(l["C"]))
        l.setdefault("v", np.zeros_like(l["C"]))
        l["C"], l["m"], l["v"] = optim.adam_step(l["C"], l["m"], l["v"], gz, LR, 0.9, 0.999, 1e-8, t)


def _oracle_mlp(weights, n_tok):
    """The oracle's inputs for ZO steps of the MLP block on n_tok tokens (fp64), outside any timing."""
    import numpy as np
    import torch
    from synth import lowrank_activations, normal, random_orthonormal
    lay = [dict(W=W, U=random_orthonormal(W.shape[1], 16, 90 + i).double().numpy(),
                C=np.zeros((W.shape[0], 16)), layer_id=i) for i, W in enumerate(weights)]
    x, _ = lowrank_activations(n_tok, 4096, 64, 0.05, 77, "cpu")
    tgt = normal((n_tok, 4096), 78, "cpu", dtype=torch.bfloat16)
    return lay, x.double().numpy(), tgt.double().numpy()


def _blas_threads():
    """Threads of numpy's BLAS (the oracle's matrix products): threadpoolctl's count where it is installed,
    else the host's cores (OpenBLAS's default)."""
    try:
        from threadpoolctl import threadpool_info
        n = [i["num_threads"] for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return max(n)
    except Exception:
        pass
    return os.cpu_count()


def _stack_names(kind):
    return ["q", "k", "v", "o", "gate", "up", "down"] if kind == "llama" else ["q", "k", "v", "o", "fc1", "fc2"]


def _oracle_decoder(w, weights, n_tok):
    """The oracle's inputs for one full-width decoder layer of a stack (a later decoder: its input holds
    both signs' activations, [2 n_tok, d]), outside any timing.  weights: name -> fp64 W."""
    import numpy as np
    from synth import lowrank_activations, random_orthonormal
    dl = {nm: dict(W=W, U=random_orthonormal(W.shape[1], w.r, 90 + i).double().numpy(),
                   C=np.zeros((W.shape[0], w.r)), layer_id=7 + i) for i, (nm, W) in enumerate(weights.items())}
    x, _ = lowrank_activations(2 * n_tok, w.d_model, 64, 0.05, 77, "cpu")
    return dl, x.double().numpy()


def _oracle_decoder_step(w, dl, x, seed, query, t):
    """One decoder's share of a ZO step: its pair forwards with the glue, then its layers' Adam updates with
    the estimator scalar of the loss pair on its output.  Returns seconds of (decoder, loss)."""
    import numpy as np
    from oracle import graphs, loss as oloss, optim, philox
    t0 = time.time()
    Y = graphs.stack_forward([dl], x, w.eps, seed, query, w.kind, store=w.act_dtype, first=False)
    t1 = time.time()
    _, _, _, a = oloss.loss_pair(Y, x.shape[0] // 2, None, w.eps)
    t2 = time.time()
    for l in dl.values():
        gz = optim.zo_gradient(a, philox.perturbation(seed, l["layer_id"], query, *l["C"].shape))
        l.setdefault("m", np.zeros_like(l["C"]))
        l.setdefault("v", np.zeros_like(l["C"]))
        l["C"], l["m"], l["v"] = optim.adam_step(l["C"], l["m"], l["v"], gz, LR, 0.9, 0.999, 1e-8, t)
    t3 = time.time()
    return (t1 - t0) + (t3 - t2), t2 - t1


def _time_decoders(w, dl, x, n_steps, t0_step=1):
    """Extrapolated seconds per full ZO step from n_steps timed decoder steps: n_decoder decoders plus one
    loss pair."""
    dec, loss = [], []
    for i in range(n_steps):
        d, l = _oracle_decoder_step(w, dl, x, 5, i + t0_step, i + t0_step)
        dec.append(d)
        loss.append(l)
    return w.n_decoder * statistics.mean(dec) + statistics.mean(loss)


def cpu_baseline(step, w, budget_s=20.0):
    """The oracle (as it stands) on the host cores.  MLP block: whole ZO steps on a 256-token sample.  Stacks:
    one full-width decoder layer (its linears, glue and Adam updates) on a 256-token sample, timed and scaled
    to the workload's decoder count (extrapolated)."""
    import torch
    n64 = lambda t: t.detach().cpu().double().numpy()
    n_tok = 256
    if w.kind == "llama_mlp":
        lay, x, tgt = _oracle_mlp([n64(step.by_name[n].W) for n in ("gate", "up", "down")], n_tok)
        t0 = time.time()
        _oracle_step(lay, x, tgt, 5, 0, 1)
        one = time.time() - t0
        reps = max(1, min(20, int(budget_s / max(one, 1e-3)) - 1))
        t0 = time.time()
        for i in range(reps):
            _oracle_step(lay, x, tgt, 5, i + 1, i + 2)
        dt = (time.time() - t0) / reps
        return {"value": n_tok / dt, "unit": UNIT, "cores": _blas_threads(), "kind": "oracle",
                "sample": f"{reps} ZO steps of the full-width Llama MLP block on {n_tok} tokens "
                          f"(numpy fp64, default BLAS threads); {dt:.3f} s per step"}
    from oracle import layers as olayers
    weights = {}
    later = 1 if w.n_decoder > 1 else 0              # a decoder past the first (input not shared) where there is one
    for nm in _stack_names(w.kind):
        lin = step.by_name[f"{later}.{nm}"]
        if lin.w_scales is not None:
            weights[nm] = olayers.dequant_int4_g128(lin.W.cpu().numpy(), lin.w_scales.float().cpu().numpy(),
                                                    lin.d_in)
        else:
            weights[nm] = n64(lin.W)
    dl, x = _oracle_decoder(w, weights, n_tok)
    t0 = time.time()
    _oracle_decoder_step(w, dl, x, 5, 0, 1)
    one = time.time() - t0
    reps = max(1, min(10, int(budget_s / max(one, 1e-3)) - 1))
    dt = _time_decoders(w, dl, x, reps, 2)
    return {"value": n_tok / dt, "unit": UNIT, "cores": _blas_threads(), "kind": "oracle",
            "extrapolated": True,
            "sample": f"{reps} timed ZO-step shares of one full-width decoder layer ({len(dl)} linears, glue, "
                      f"Adam) of {w.name} on {n_tok} tokens per perturbation (numpy fp64, default BLAS "
                      f"threads), scaled to {w.n_decoder} decoders plus one loss pair (extrapolated): "
                      f"{dt:.2f} s per full step"}


def run_reference(args):
    """The CPU oracle as the reference arm: --steps timed steps, each one full-width decoder layer's share of
    a ZO step of the default workload on a bounded token sample, reported as the extrapolated full step."""
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if rank != 0:
        return
    import torch
    from synth import workload, normal, tensor_seed
    w = workload(DEFAULT_WORKLOAD)
    n_tok = args.ref_tokens
    dims = {s.name.split(".")[1]: (s.d_out, s.d_in) for s in w.linears() if s.name.startswith("1.")}
    # the weights drawn on the CPU with the same shapes (the reference arm never touches the GPU)
    weights = {nm: normal(dims[nm], tensor_seed(w, "W", f"1.{nm}"), "cpu", std=w.weight_std,
                          dtype=torch.bfloat16).double().numpy() for nm in _stack_names(w.kind)}
    dl, x = _oracle_decoder(w, weights, n_tok)
    for i in range(args.warmup):
        _oracle_decoder_step(w, dl, x, 5, i + 1, i + 1)
    dt = _time_decoders(w, dl, x, args.steps, args.warmup + 1)
    v = n_tok / dt
    sample = (f"{args.steps} timed ZO-step shares of one full-width decoder layer of {w.name} on {n_tok} tokens "
              f"per perturbation (numpy fp64), scaled to {w.n_decoder} decoders plus one loss pair "
              f"(extrapolated)")
    print(json.dumps({
        "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": dt * 1e3, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f64", "data": "synthetic", "impl": "reference",
        "config": {"workload": DEFAULT_WORKLOAD, "tokens_per_perturbation": n_tok, "r": w.r, "eps": w.eps,
                   "adapted_linears": len(w.linears())},
        "cpu_baseline": {"value": v, "unit": UNIT, "cores": _blas_threads(), "kind": "oracle",
                         "sample": sample, "extrapolated": True},
        "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD,
                    choices=["llama_mlp_bf16", "llama_stack_bf16", "llama_stack_int4", "opt_stack_fp16"])
    ap.add_argument("--tokens", type=int, default=None, help="tokens per perturbation (default: the workload's)")
    ap.add_argument("--queries", type=int, default=None,
                    help="one-sided estimator with this many queries (Algorithm 2); default: two-sided pair")
    ap.add_argument("--rank", type=int, default=None, help="basis rank r (default: the workload's; 1..256)")
    ap.add_argument("--decoders", type=int, default=None,
                    help="stacks only: fewer decoder layers (profiling captures of a few GB; not a bench workload)")
    ap.add_argument("--diag", action="store_true", help="also time the Section 5.3 subspace diagnostics")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--soak", type=float, default=2.0,
                    help="seconds of untimed steps before the timed region (clocks reach their loaded state)")
    ap.add_argument("--cpu-budget", type=float, default=20.0, help="seconds of oracle work for cpu_baseline")
    ap.add_argument("--ref-tokens", type=int, default=64, help="tokens per oracle step in the reference arm")
    ap.add_argument("--measure-peak", choices=["fp16", "bf16"], default=None,
                    help="only measure the dense tensor peak of this dtype (torch.matmul 8192^3) and exit")
    ap.add_argument("--measure-read", action="store_true",
                    help="only time reads of 50 MB to 805 MB (zoact_loss_pair, the projection, torch.sum) and exit")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.measure_peak:
        measure_peak(args.measure_peak)
    elif args.measure_read:
        measure_read()
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
