#!/usr/bin/env python
"""ZO-step throughput of the ZO-Act hot path on GB300.

Workload (default): the Llama-3-8B MLP block in bf16 -- gate/up 4096 -> 14336
on a shared input, SiLU gate, down 14336 -> 4096 -- r = 16, T = 2048 tokens per
perturbation (4096 stacked rows for the +/- pair), MSE to N(0,1) targets,
eps = 1e-3, Adam on all coefficients.  Synthetic data: rank-64 Gaussian signal
plus 5% noise, unit RMS per token; W ~ N(0, 0.02); bases from a 2048-token
calibration batch (Algorithm 1, on the device, before timing).

One step = zoact_lowrank_proj + zoact_pair_forward_gated (gate/up) +
zoact_lowrank_proj + zoact_pair_forward (down) + zoact_loss_pair +
zoact_adam_step, all on one stream, no host synchronisation.

value = training tokens/s = world_size * T / step time (device time, CUDA
events around exactly --steps steps, max over ranks).  The weights (352 MB) are
larger than L2 (129 MB), so every step streams them from HBM.
`--impl reference` times the CPU oracle (numpy fp64) on a bounded sample of the
same workload instead.
"""
import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "ZO-step tokens/s per adapted-linear stack; % of HBM or tensor-pipe roofline"
UNIT = "tokens/s"
T_TOKENS = 2048
D_MODEL, D_FF, RANK = 4096, 14336, 16
N_CAL = 2048
EPS = 1e-3
LR = 1e-4


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p["hbm_gbs"], p["bf16_tflops"], p["bf16_tflops_sustained"], "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 100 ms in a child process."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = os.path.join(ROOT, "gpurun_out", f"clocks_gpu{index}.csv")

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


def build_mlp(ctx, dev, rank, seed=0):
    """Weights, bases and the ZOStep of the Llama MLP block (inputs per rank for weak scaling)."""
    import torch
    import paper_2607_01125_gb300 as zo
    from paper_2607_01125_gb300.model import AdaptedLinear, ZOStep
    from synth import workload, normal, lowrank_activations, tensor_seed
    w = workload("llama_mlp_bf16", seed=seed)
    x_all, _ = lowrank_activations(N_CAL + T_TOKENS, D_MODEL, 64, 0.05, tensor_seed(w, "x", rank), dev)
    X_cal, x = x_all[:N_CAL].contiguous(), x_all[N_CAL:].contiguous()
    target = normal((T_TOKENS, D_MODEL), tensor_seed(w, "target", rank), dev, dtype=torch.bfloat16)
    Wg = normal((D_FF, D_MODEL), tensor_seed(w, "W", "gate"), dev, std=w.weight_std, dtype=torch.bfloat16)
    Wu = normal((D_FF, D_MODEL), tensor_seed(w, "W", "up"), dev, std=w.weight_std, dtype=torch.bfloat16)
    Wd = normal((D_MODEL, D_FF), tensor_seed(w, "W", "down"), dev, std=w.weight_std, dtype=torch.bfloat16)
    # Algorithm 1: one calibration pass of the base model, bases of each layer's input
    U_x = torch.empty(D_MODEL, RANK, device=dev)
    zo.zoact_basis_init(ctx, X_cal, RANK, U_x, oversample=16, n_iter=8, seed=tensor_seed(w, "basis", "x"))
    C0 = torch.zeros(D_FF * RANK, device=dev)
    Hc = torch.empty(2 * N_CAL, D_FF, dtype=torch.bfloat16, device=dev)
    zo.zoact_pair_forward_gated(ctx, zo.make_layer(Wg, U_x, C0, 0), zo.make_layer(Wu, U_x, C0, 1), X_cal, N_CAL,
                                True, 0.0, 0, 0, Hc)
    U_h = torch.empty(D_FF, RANK, device=dev)
    zo.zoact_basis_init(ctx, Hc[:N_CAL].contiguous(), RANK, U_h, oversample=16, n_iter=8,
                        seed=tensor_seed(w, "basis", "h"))
    del Hc
    lins = [AdaptedLinear("gate", Wg, U_x, 0, 0, RANK), AdaptedLinear("up", Wu, U_x, 1, D_FF * RANK, RANK),
            AdaptedLinear("down", Wd, U_h, 2, 2 * D_FF * RANK, RANK)]
    step = ZOStep(ctx, "llama_mlp", lins, T_TOKENS, "bf16", eps=EPS, lr=LR)
    return step, x, target


class MLPRunner:
    """One ZO step of the MLP block with the tensor-core launches bracketed by CUDA events."""

    def __init__(self, step, world):
        import torch
        import paper_2607_01125_gb300 as zo
        self.zo, self.torch = zo, torch
        self.s = step
        self.world = world
        T = step.T
        dev = step.device
        self.P_x = torch.empty(T, RANK, device=dev)
        self.P_h = torch.empty(2 * T, RANK, device=dev)
        self.H = torch.empty(2 * T, D_FF, dtype=torch.bfloat16, device=dev)
        self.Y = torch.empty(2 * T, D_MODEL, dtype=torch.bfloat16, device=dev)
        self.events = []

    def run(self, x, target, t, seed, instrument):
        zo, torch, s = self.zo, self.torch, self.s
        g, u, d = s.by_name["gate"], s.by_name["up"], s.by_name["down"]
        zo.zoact_lowrank_proj(s.ctx, x, g.U, self.P_x)                 # gate and up share U (same input)
        if instrument:
            e0 = torch.cuda.Event(enable_timing=True); e0.record()
        zo.zoact_pair_forward_gated(s.ctx, g.layer, u.layer, x, s.T, True, s.eps, seed, t, self.H,
                                    P_gate=self.P_x, P_up=self.P_x)
        if instrument:
            e1 = torch.cuda.Event(enable_timing=True); e1.record()
        zo.zoact_lowrank_proj(s.ctx, self.H, d.U, self.P_h)
        if instrument:
            e2 = torch.cuda.Event(enable_timing=True); e2.record()
        zo.zoact_pair_forward(s.ctx, d.layer, self.H, s.T, False, s.eps, seed, t, self.Y, P=self.P_h)
        if instrument:
            e3 = torch.cuda.Event(enable_timing=True); e3.record()
            self.events.append((e0, e1, e2, e3))
        s.loss(self.Y, target)
        if self.world > 1:
            from paper_2607_01125_gb300.dp import allreduce_loss
            allreduce_loss(s.loss_out)           # L+, L-, D and a are means over equal token counts
        s.update(t, seed, t)
        return s.loss_out


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
    step, x, target = build_mlp(ctx, dev, rank)
    runner = MLPRunner(step, world)
    seed = 1234

    def barrier():
        if world > 1:
            dist.barrier()

    # warm-up (untimed), then a ~2 s soak so clocks are at their loaded steady state
    t = 1
    for _ in range(args.warmup):
        runner.run(x, target, t, seed, False); t += 1
    sampler = ClockSampler(local)
    sampler.start()
    torch.cuda.synchronize()
    soak_end = time.time() + args.soak
    while time.time() < soak_end:
        for _ in range(20):
            runner.run(x, target, t, seed, False); t += 1
        torch.cuda.synchronize()

    # ---- timed region: exactly args.steps steps ----
    n0 = ctx.launch_count()
    barrier(); torch.cuda.synchronize()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.nvtx.range_push("timed")          # profilers select the timed steps by this range
    start.record()
    for _ in range(args.steps):
        runner.run(x, target, t, seed, True); t += 1
    end.record()
    torch.cuda.nvtx.range_pop()
    torch.cuda.synchronize(); barrier()
    launches = ctx.launch_count() - n0
    ms = start.elapsed_time(end) / args.steps
    gemm_ms = [(a.elapsed_time(b), c.elapsed_time(d)) for a, b, c, d in runner.events]

    # ---- end to end through the public API with host buffers ----
    x_h = x.cpu().pin_memory()
    t_h = target.cpu().pin_memory()
    out_h = torch.empty(4, dtype=torch.float64).pin_memory()
    x_d, t_d = torch.empty_like(x), torch.empty_like(target)
    barrier(); torch.cuda.synchronize()
    e_s, e_e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e_s.record()
    for _ in range(args.steps):
        x_d.copy_(x_h, non_blocking=True)
        t_d.copy_(t_h, non_blocking=True)
        out = runner.run(x_d, t_d, t, seed, False); t += 1
        out_h.copy_(out, non_blocking=True)
    e_e.record()
    torch.cuda.synchronize(); barrier()
    clocks = sampler.stop()
    e2e_ms = e_s.elapsed_time(e_e) / args.steps
    status = ctx.device_status()

    if world > 1:
        tt = torch.tensor([ms, e2e_ms], device=dev)
        dist.all_reduce(tt, op=dist.ReduceOp.MAX)
        ms, e2e_ms = float(tt[0]), float(tt[1])
    if rank != 0:
        return
    hbm, tf_burst, tf_sust, peak_kind = _peaks()
    T = T_TOKENS
    flops_gated = 2.0 * T * D_MODEL * (2 * D_FF)          # gate + up on T shared rows
    flops_down = 2.0 * (2 * T) * D_FF * D_MODEL            # down on 2T stacked rows
    tg = statistics.mean(a for a, _ in gemm_ms)
    td = statistics.mean(b for _, b in gemm_ms)
    achieved = (flops_gated + flops_down) / ((tg + td) * 1e-3) / 1e12
    line = {
        "metric": METRIC, "value": world * T / (ms * 1e-3), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": "llama_mlp_bf16", "tokens_per_perturbation": T, "stacked_rows": 2 * T,
                   "d_model": D_MODEL, "d_ff": D_FF, "r": RANK, "eps": EPS, "estimator": "two-sided, q=1",
                   "l2": "inputs larger than L2 (352 MB of frozen weights streamed per step)",
                   "parallelism": f"dp{world}" if world > 1 else "single"},
        "evaluated_tokens_per_s": world * 2 * T / (ms * 1e-3),
        "zo_steps_per_s": 1e3 / ms,
        "kernel_ms": {"pair_forward_gated": tg, "pair_forward_down": td},
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": tf_burst, "unit": "TFLOP/s",
                     "frac": achieved / tf_burst, "peak_kind": f"bf16 dense burst, {peak_kind}",
                     "kernel": "pair_tc_kernel (gated gate/up + down)",
                     "traffic": None},
        "e2e": {"value": world * T / (e2e_ms * 1e-3), "unit": UNIT,
                "h2d_bytes_per_step": x.numel() * 2 + target.numel() * 2, "d2h_bytes_per_step": 32},
        "gpu_launches": launches,
        "clocks": clocks,
        "device_status": status,
    }
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(step, budget_s=args.cpu_budget)
    print(json.dumps(line))


def _oracle_sample_step(step, n_tok, seed):
    """Everything the oracle needs for one ZO step on n_tok tokens (fp64 numpy), prepared outside the timing."""
    import numpy as np
    from synth import lowrank_activations, normal, random_orthonormal
    n64 = lambda t: t.detach().double().cpu().numpy()
    g, u, d = step.by_name["gate"], step.by_name["up"], step.by_name["down"]
    lay = [dict(W=n64(l.W), U=random_orthonormal(l.d_in, RANK, 90 + i).double().numpy(),
                C=np.zeros((l.d_out, RANK)), layer_id=l.layer_id) for i, l in enumerate((g, u, d))]
    x, _ = lowrank_activations(n_tok, D_MODEL, 64, 0.05, seed, "cpu")
    tgt = normal((n_tok, D_MODEL), seed + 1, "cpu", dtype=__import__("torch").bfloat16)
    return lay, x.double().numpy(), tgt.double().numpy()


def _oracle_step(lay, x, tgt, seed, query, t):
    import numpy as np
    from oracle import graphs, loss as oloss, optim, philox
    Y = graphs.llama_mlp_forward(lay, x, EPS, seed, query, store="bf16")
    _, _, _, a = oloss.loss_pair(Y, x.shape[0], tgt, EPS)
    for l in lay:
        gz = optim.zo_gradient(a, philox.perturbation(seed, l["layer_id"], query, *l["C"].shape))
        l.setdefault("m", np.zeros_like(l["C"]))
        l.setdefault("v", np.zeros_like(l["C"]))
        l["C"], l["m"], l["v"] = optim.adam_step(l["C"], l["m"], l["v"], gz, LR, 0.9, 0.999, 1e-8, t)


def cpu_baseline(step, budget_s=20.0, n_tok=None):
    """The oracle (as it stands) on the host cores: ZO steps of the same block on a token sample."""
    n_tok = n_tok or 256
    lay, x, tgt = _oracle_sample_step(step, n_tok, 77)
    t0 = time.time()
    _oracle_step(lay, x, tgt, 5, 0, 1)
    one = time.time() - t0
    reps = max(1, min(20, int(budget_s / max(one, 1e-3)) - 1))
    t0 = time.time()
    for i in range(reps):
        _oracle_step(lay, x, tgt, 5, i + 1, i + 2)
    dt = (time.time() - t0) / reps
    return {"value": n_tok / dt, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"{reps} ZO steps of the full-width Llama MLP block on {n_tok} tokens "
                      f"(numpy fp64, default BLAS threads); {dt:.3f} s per step"}


def run_reference(args):
    """The CPU oracle as the reference arm: --steps timed ZO steps on a bounded token sample."""
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if rank != 0:
        return
    import torch
    import numpy as np
    from synth import workload, normal, tensor_seed, lowrank_activations, random_orthonormal
    w = workload("llama_mlp_bf16")
    n_tok = args.ref_tokens
    # weights drawn on the CPU with the same shapes (the reference arm never touches the GPU)
    shapes = [("gate", D_FF, D_MODEL), ("up", D_FF, D_MODEL), ("down", D_MODEL, D_FF)]
    lay = []
    for i, (nm, do, di) in enumerate(shapes):
        Wt = normal((do, di), tensor_seed(w, "W", nm), "cpu", std=w.weight_std, dtype=torch.bfloat16)
        lay.append(dict(W=Wt.double().numpy(), U=random_orthonormal(di, RANK, 90 + i).double().numpy(),
                        C=np.zeros((do, RANK)), layer_id=i))
    x, _ = lowrank_activations(n_tok, D_MODEL, 64, 0.05, 77, "cpu")
    x = x.double().numpy()
    tgt = normal((n_tok, D_MODEL), 78, "cpu", dtype=torch.bfloat16).double().numpy()
    t = 1
    for _ in range(args.warmup):
        _oracle_step(lay, x, tgt, 5, t, t); t += 1
    t0 = time.time()
    for _ in range(args.steps):
        _oracle_step(lay, x, tgt, 5, t, t); t += 1
    dt = (time.time() - t0) / args.steps
    v = n_tok / dt
    sample = f"{args.steps} ZO steps of the full-width Llama MLP block on {n_tok} tokens (numpy fp64)"
    print(json.dumps({
        "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": dt * 1e3, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f64", "data": "synthetic", "impl": "reference",
        "config": {"workload": "llama_mlp_bf16", "tokens_per_perturbation": n_tok, "d_model": D_MODEL,
                   "d_ff": D_FF, "r": RANK, "eps": EPS},
        "cpu_baseline": {"value": v, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle", "sample": sample},
        "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--soak", type=float, default=2.0,
                    help="seconds of untimed steps before the timed region (clocks reach their loaded state)")
    ap.add_argument("--cpu-budget", type=float, default=20.0, help="seconds of oracle work for cpu_baseline")
    ap.add_argument("--ref-tokens", type=int, default=64, help="tokens per oracle step in the reference arm")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
