#!/usr/bin/env python3
"""Dream-rollout throughput on GB300: env-steps/s of wm_rollout, with its roofline.

One "step" is one wm_rollout call over the whole workload: T dream steps of B
independent episodes (controller, mask + action choice, LSTM, mixture head,
sampling, reward / done).  Default workload: the large-batch tensor-core
regime, B=65536 episodes x T=64 steps, Z=128, A=512 (10% valid mask), H=1024,
K=8, bf16 operands / fp32 state, sampled controller at temperature 1
(``synth.WORKLOADS['large_bf16']``), the largest configuration that fits one GPU.
For workloads whose episodes end (done head or NO-OP), ``value`` counts live
(episode, step) pairs only; frozen pairs are executed but not counted.

Timing: W untimed warm-ups, then K steps each bracketed by CUDA events on the
launching stream, with a 512 MiB write between steps to flush the 129 MB L2.
N GPUs (torchrun): every rank runs its own B episodes (episode_offset =
rank * B), no data-path collective, max time over ranks -> weak scaling.

``--impl reference`` times the CPU oracle (the plain C definition of the same
steps) on the host cores instead, on a bounded sample of the same workload.
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

import synth  # noqa: E402

CLOCK_Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
           "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
           "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


def flops_per_env_step(cfg: dict) -> float:
    """Algorithmic FLOPs of one (episode, step): the three contractions plus heads.

    controller [Z+H] x [Z+H, A], gates [Z+H] x [Z+H, 4H] (the one-hot action
    row is a gather, not FLOPs), mixture head [H] x [H, 3KZ], reward and done.
    """
    Z, A, H, K = cfg["z_dim"], cfg["a_dim"], cfg["h_dim"], cfg["k_mix"]
    return 2.0 * ((Z + H) * A + (Z + H) * 4 * H + H * 3 * K * Z + 2 * H)


def load_peaks() -> dict:
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


def fp32_simt_peak_tflops() -> float:
    # 152 SMs x 128 fp32 FMA lanes x 2 FLOP x 2.07 GHz (maximum SM clock)
    return 152 * 128 * 2 * 2.07e9 / 1e12


# kernel class -> (kernel as the profiler names it, source file)
KERNELS = {"fused": ("k_fused", "wm_fused.cu"),
           "fused_small": ("k_small", "wm_small.cu"),
           "tc_ctrl": ("k_tc_gemm<EpiCtrl>", "wm_tensor.cu"),
           "tc_gates": ("k_tc_gemm<EpiGates>", "wm_tensor.cu"),
           "tc_heads": ("k_tc_gemm<EpiHeads>", "wm_tensor.cu"),
           "step_gemm": ("k_gemm", "wm_step.cu"),
           "step_cell": ("k_select_cell", "wm_step.cu"),
           "step_sample": ("k_sample", "wm_step.cu")}


def nll_flops_per_step(cfg: dict) -> float:
    """Algorithmic FLOPs of one teacher-forced (sequence, step): gates and mixture head."""
    Z, H, K = cfg["z_dim"], cfg["h_dim"], cfg["k_mix"]
    return 2.0 * ((Z + H) * 4 * H + H * (3 * K * Z + 2))


def nll_inputs(cfg: dict, rank: int = 0):
    """(z_seq, actions) of the scoring workload; rank r scores its own sequences."""
    w = synth.WORKLOADS["nll"]
    return synth.teacher_inputs(w["N"], w["T"], cfg["z_dim"], cfg["a_dim"], seed=rank)[:2]


def kernel_flops(cls: str, cfg: dict, B: int, T: int, launches: int) -> float:
    """Algorithmic FLOPs of one launch of a kernel class (its contraction)."""
    Z, A, H, K = cfg["z_dim"], cfg["a_dim"], cfg["h_dim"], cfg["k_mix"]
    if cls in ("fused", "fused_small"):
        return (nll_flops_per_step(cfg) if cfg.get("teacher") else flops_per_env_step(cfg)) * B * T
    if cls == "tc_ctrl":
        return 2.0 * B * (Z + H) * A
    if cls == "tc_gates":
        return 2.0 * B * (Z + H) * 4 * H
    if cls == "tc_heads":
        return 2.0 * B * H * (3 * K * Z + 2)
    if cls == "step_gemm":  # two GEMMs per step: gates (+ controller), then heads
        return 2.0 * B * ((Z + H) * (4 * H + (0 if cfg.get("teacher") else A)) + H * (3 * K * Z + 2)) / 2
    return 0.0


def kernel_source_sha(src: str) -> str:
    with open(os.path.join(ROOT, "paper_2205_01435_gb300", "csrc", src), "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def ncu_traffic(kernel_key: str, sha: str):
    """DRAM bytes per launch from a committed ncu capture of this exact kernel source."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    e = d.get(kernel_key)
    if not e or e.get("source_sha") != sha:
        return None
    return e.get("dram_bytes_per_launch")


class ClockSampler:
    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            self.path = f"/tmp/wm_clocks_{os.getpid()}.csv"
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={CLOCK_Q}",
                 "--format=csv,noheader,nounits", "-lms", "100"], stdout=self.f,
                stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.f.close()

    def summary(self) -> dict:
        if self.proc is None or not self.path or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax = float(parts[2])
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax,
                "reasons": sorted(reasons), "samples": len(sm)}


def max_over_ranks(value: float, ws: int, device=None) -> float:
    """The maximum of a per-rank value over all ranks (the slowest rank's time)."""
    import torch
    import torch.distributed as dist

    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    if ws > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(value: float, ws: int, device=None) -> float:
    """The sum of a per-rank count over all ranks."""
    import torch
    import torch.distributed as dist

    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    if ws > 1:
        dist.all_reduce(t)
    return float(t.item())


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def measure_e2e(model, z0, mask, T, ep0, args, flush, dev, ws, B, cfg, env_steps, shaping=None,
                loc_mask=None):
    """The same rollout through the C ABI with pinned HOST arrays: copies are timed.
    env_steps: the (episode, step) pairs one call counts over all ranks."""
    import torch

    sh = {} if shaping is None else {"rt0": torch.from_numpy(shaping[0]).pin_memory(),
                                     "mem0": torch.from_numpy(shaping[1]).pin_memory()}
    if loc_mask is not None:
        sh["loc_mask"] = torch.from_numpy(loc_mask).pin_memory()
    zh = torch.from_numpy(z0).pin_memory()
    mh = torch.from_numpy(mask).pin_memory()
    hout = {"z": torch.empty((T + 1, B, cfg["z_dim"]), pin_memory=True),
            "actions": torch.empty((T, B), dtype=torch.int32, pin_memory=True),
            "rewards": torch.empty((T, B), pin_memory=True),
            "done": torch.empty((T, B), dtype=torch.uint8, pin_memory=True)}
    for _ in range(2):
        model.rollout(zh, T, mask=mh, episode_offset=ep0, want_final=False, out=hout, **sh)
    torch.cuda.synchronize()
    e2e_t = []
    for i in range(args.steps):
        flush.fill_(float(i))
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        model.rollout(zh, T, mask=mh, episode_offset=ep0, want_final=False, out=hout, **sh)
        e2e_t.append(time.perf_counter() - t0)
    e2e_value = env_steps / max_over_ranks(sum(e2e_t) / len(e2e_t), ws, dev)
    h2d = zh.numel() * 4 + mh.numel() * 4 + sum(v.numel() * 4 for v in sh.values())
    d2h = sum(v.numel() * v.element_size() for v in hout.values())

    return e2e_value, h2d, d2h


def kernel_timing_pass(model, step, flush, stream, steps: int) -> dict:
    import torch

    torch.cuda.synchronize()
    model.set_timing(True)
    for i in range(steps):
        flush.fill_(float(i))
        step()
    torch.cuda.synchronize()
    kt = model.kernel_times()
    model.set_timing(False)
    return kt


def run_nll(args) -> None:
    """Teacher-forced scoring (wm_mdn_nll) of the nll workload: scored (sequence, step)
    pairs per second, same timing, e2e, roofline and CPU-baseline rules as the rollouts."""
    import torch

    import paper_2205_01435_gb300 as pkg

    ws, rank, local = dist_env()
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    wm = pkg.load()
    cfg = synth.model_config("nll", precision=args.precision or "bf16")
    if args.path:
        cfg["path"] = args.path
    w = synth.weights(cfg)
    zs, acts = nll_inputs(cfg, rank)
    T, N = acts.shape
    model = wm.WorldModel(cfg, w, device=local)
    dev = torch.device("cuda", local)
    zc, ac = torch.from_numpy(zs).to(dev), torch.from_numpy(acts).to(dev)
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    for _ in range(args.warmup):
        model.mdn_nll(zc, ac, stream=stream)
    torch.cuda.synchronize()
    path_name, launches = model.last_path, model.last_launches
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    with ClockSampler(local) as clk:
        for i in range(args.steps):
            flush.fill_(float(i))
            ev[i][0].record(stream)
            model.mdn_nll(zc, ac, stream=stream)
            ev[i][1].record(stream)
        torch.cuda.synchronize()
    kt = kernel_timing_pass(model, lambda: model.mdn_nll(zc, ac, stream=stream), flush, stream, args.steps)
    ms_per_step = max_over_ranks(sum(a.elapsed_time(b) for a, b in ev), ws, dev) / args.steps
    value = N * T * ws / (ms_per_step / 1e3)
    # e2e: pinned host inputs and output
    zh, ah = torch.from_numpy(zs).pin_memory(), torch.from_numpy(acts).pin_memory()
    model.mdn_nll(zh, ah)
    e2e_t = []
    for i in range(args.steps):
        flush.fill_(float(i))
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        r = model.mdn_nll(zh, ah)
        e2e_t.append(time.perf_counter() - t0)
    e2e_value = N * T * ws / max_over_ranks(sum(e2e_t) / len(e2e_t), ws, dev)
    peaks = load_peaks()
    tcfg = dict(cfg, teacher=1)
    timed = {k: v for k, v in kt.items() if k in KERNELS}
    dom = max(timed, key=lambda k: timed[k][0])
    dom_ms, dom_n = timed[dom]
    fl = kernel_flops(dom, tcfg, N, T, dom_n)
    achieved = fl / (dom_ms / dom_n / 1e3) / 1e12
    if cfg["precision"] == "bf16" and dom in ("fused", "tc_gates", "tc_heads"):
        bound, peak, psrc = "tensor", peaks["bf16_tflops"], peaks["source"] + " bf16 burst"
    elif dom in ("tc_gates", "tc_heads"):  # fp32 on the tensor cores: three bf16 passes
        bound, peak = "tensor", peaks["bf16_tflops"] / 3
        psrc = peaks["source"] + " bf16 burst / 3 (fp32 products as three bf16 passes)"
    else:
        bound, peak, psrc = "alu", fp32_simt_peak_tflops(), "derived: 152 SM x 128 fp32 FMA x 2 FLOP x 2.07 GHz"
    kname, ksrc = KERNELS[dom]
    call_fl = nll_flops_per_step(cfg) * N * T
    roof = {"bound": bound, "achieved": round(achieved, 3), "peak": round(peak, 1), "unit": "TFLOP/s",
            "frac": round(achieved / peak, 5),
            "traffic": ncu_traffic(f"{kname}/nll_{cfg['precision']}", kernel_source_sha(ksrc)),
            "peak_source": psrc, "kernel": f"{kname}/nll_{cfg['precision']}",
            "launch_ms": round(dom_ms / dom_n, 5), "launches": dom_n, "algorithmic_flops_per_launch": fl,
            "kernel_shares": {k: round(v[0] / sum(x[0] for x in kt.values()), 4) for k, v in sorted(kt.items())},
            "call_frac_of_tensor_roofline": round(call_fl / (ms_per_step / 1e3) / 1e12 / peaks["bf16_tflops"], 5)}
    line = {"metric": "teacher-forced scored steps/s (wm_mdn_nll)", "value": round(value, 1),
            "unit": "scored-steps/s", "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(ms_per_step, 4), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16" if cfg["precision"] == "bf16" else "f32",
            "data": "synthetic (seeded: weights N(0,0.05^2), z ~ N(0,1), actions uniform)",
            "config": {"workload": f"nll_{cfg['precision']}", "N": N, "T": T, "z": cfg["z_dim"],
                       "A": cfg["a_dim"], "H": cfg["h_dim"], "K": cfg["k_mix"], "kernel_path": path_name,
                       "l2": "flushed between timed steps (512 MiB write)",
                       "parallelism": f"sequences sharded over {ws} GPU(s), no collective"},
            "e2e": {"value": round(e2e_value, 1), "unit": "scored-steps/s",
                    "h2d_bytes_per_step": zh.numel() * 4 + ah.numel() * 4, "d2h_bytes_per_step": N * 4},
            "gpu_launches": launches * args.steps, "roofline": roof, "clocks": clk.summary()}
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        import oracle
        n = max(8, min(N, args.cpu_episodes or N // 4))
        threads = os.cpu_count() or 1
        t0 = time.perf_counter()
        oracle.mdn_nll(cfg, w, zs[:, :n], acts[:, :n], nthreads=threads)
        dt = time.perf_counter() - t0
        line["cpu_baseline"] = {"value": round(n * T / dt, 2), "unit": "scored-steps/s", "cores": threads,
                                "kind": "oracle", "sample": f"{n} of {N} sequences x {T} steps, {threads} threads, {dt:.1f} s"}
    if rank == 0:
        print(json.dumps(line), flush=True)
    model.close()


def train_flops_per_step(cfg: dict) -> float:
    """Algorithmic FLOPs of one (sequence, step) of the training step: the forward's gates and
    head, then the backward's gate recompute, dY = dMD W_mdn^T, the recurrent dG W_h^T and
    the weight gradients X^T dG and Y^T dMD."""
    Z, H, K = cfg["z_dim"], cfg["h_dim"], cfg["k_mix"]
    KX, M = Z + H, 3 * K * Z
    fwd = 2.0 * (KX * 4 * H + H * (M + 2))
    bwd = 2.0 * (KX * 4 * H + M * H + 4 * H * H + KX * 4 * H + H * M)
    return fwd + bwd


def run_train(args) -> None:
    """The world model's training step (wm_mdn_nll_backward) on the nll workload: loss and
    gradient of 512 sequences x 128 steps, in scored (sequence, step) pairs per second."""
    import torch

    import paper_2205_01435_gb300 as pkg

    ws, rank, local = dist_env()
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    wm = pkg.load()
    cfg = synth.model_config("nll", precision=args.precision or "bf16")
    if args.path:
        cfg["path"] = args.path
    w = synth.weights(cfg)
    zs, acts = nll_inputs(cfg, rank)
    T, N = acts.shape
    model = wm.WorldModel(cfg, w, device=local)
    dev = torch.device("cuda", local)
    zc, ac = torch.from_numpy(zs).to(dev), torch.from_numpy(acts).to(dev)
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    for _ in range(args.warmup):
        model.mdn_nll_backward(zc, ac, stream=stream)
    torch.cuda.synchronize()
    path_name, launches = model.last_path, model.last_launches
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    with ClockSampler(local) as clk:
        for i in range(args.steps):
            flush.fill_(float(i))
            ev[i][0].record(stream)
            model.mdn_nll_backward(zc, ac, stream=stream)
            ev[i][1].record(stream)
        torch.cuda.synchronize()
    kt = kernel_timing_pass(model, lambda: model.mdn_nll_backward(zc, ac, stream=stream), flush, stream,
                            args.steps)
    ms_per_step = max_over_ranks(sum(a.elapsed_time(b) for a, b in ev), ws, dev) / args.steps
    value = N * T * ws / (ms_per_step / 1e3)
    zh, ah = torch.from_numpy(zs).pin_memory(), torch.from_numpy(acts).pin_memory()
    model.mdn_nll_backward(zh, ah)
    e2e_t = []
    for i in range(args.steps):
        flush.fill_(float(i))
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        model.mdn_nll_backward(zh, ah)
        e2e_t.append(time.perf_counter() - t0)
    e2e_value = N * T * ws / max_over_ranks(sum(e2e_t) / len(e2e_t), ws, dev)
    peaks = load_peaks()
    all_ms = sum(v[0] for v in kt.values())
    call_fl = train_flops_per_step(cfg) * N * T
    bf = cfg["precision"] == "bf16"
    # fp32: the forward's products run as three bf16 passes and the backward's GEMMs on the
    # library's bf16 emulation of fp32, so the denominator is the bf16 peak / 3 (the contraction's
    # passes), as for the fp32 scoring and rollout lines
    peak = peaks["bf16_tflops"] if bf else peaks["bf16_tflops"] / 3
    achieved = call_fl / (ms_per_step / 1e3) / 1e12
    Z, A, H, K = cfg["z_dim"], cfg["a_dim"], cfg["h_dim"], cfg["k_mix"]
    grad_bytes = 4 * ((Z + A + H) * 4 * H + 4 * H + H * 3 * K * Z + 3 * K * Z)
    roof = {"bound": "tensor", "achieved": round(achieved, 3), "peak": round(peak, 1),
            "unit": "TFLOP/s", "frac": round(achieved / peak, 5), "traffic": None,
            "peak_source": (peaks["source"] + " bf16 burst") if bf else
            peaks["source"] + " bf16 burst / 3 (fp32 products as three bf16 passes)",
            "kernel": "whole training step (forward + BPTT)", "algorithmic_flops_per_step": call_fl,
            "kernel_shares": {k: round(v[0] / all_ms, 4) for k, v in sorted(kt.items())}}
    line = {"metric": "world-model training steps: scored (sequence, step) pairs/s (wm_mdn_nll_backward)",
            "value": round(value, 1), "unit": "scored-steps/s", "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(ms_per_step, 4), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if bf else "f32",
            "data": "synthetic (seeded: weights N(0,0.05^2), z ~ N(0,1), actions uniform)",
            "config": {"workload": f"nll_{cfg['precision']}_train", "N": N, "T": T, "z": Z, "A": A, "H": H,
                       "K": K, "kernel_path": path_name, "l2": "flushed between timed steps (512 MiB write)",
                       "parallelism": f"sequences sharded over {ws} GPU(s), no collective"},
            "e2e": {"value": round(e2e_value, 1), "unit": "scored-steps/s",
                    "h2d_bytes_per_step": zh.numel() * 4 + ah.numel() * 4,
                    "d2h_bytes_per_step": N * 4 + grad_bytes},
            "gpu_launches": launches * args.steps, "roofline": roof, "clocks": clk.summary()}
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        import oracle
        n = max(4, min(N, args.cpu_episodes or 16))
        threads = os.cpu_count() or 1
        t0 = time.perf_counter()
        oracle.mdn_nll_grad(cfg, w, zs[:, :n], acts[:, :n], nthreads=threads)
        dt = time.perf_counter() - t0
        line["cpu_baseline"] = {"value": round(n * T / dt, 2), "unit": "scored-steps/s", "cores": threads,
                                "kind": "oracle", "sample": f"{n} of {N} sequences x {T} steps, loss and "
                                                            f"gradient, {threads} threads, {dt:.1f} s"}
    if rank == 0:
        print(json.dumps(line), flush=True)
    model.close()


def run_ours(args) -> None:
    import torch
    import torch.distributed as dist

    import paper_2205_01435_gb300 as pkg

    ws, rank, local = dist_env()
    if ws > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    wm = pkg.load()
    name = args.workload
    # rank r runs shard r of the global batch: its own z0 and masks, Philox episodes r*B + b
    cfg, w, z0, mask, B, T = synth.rollout_inputs(name, B=args.batch, shard=rank)
    if args.path:
        cfg["path"] = args.path
    shaping = None
    if args.reward == "shaped":
        cfg["reward_mode"] = 1
        shaping = synth.shaping_state(B, shard=rank)
    if args.xfers:  # hierarchical action: NX xfers (with the NO-OP) x L = A - NX locations
        NX = args.xfers
        cfg["n_xfers"] = NX
        mask, loc_mask = synth.hier_masks(T, B, NX, cfg["a_dim"] - NX,
                                          synth.WORKLOADS[name]["mask_density"], shard=rank)
    P = args.population
    if P:
        if B % P or (B // P) % 256:
            raise SystemExit("--population: B / P must be a multiple of 256")
        cfg["value_head"] = 1
    model = wm.WorldModel(cfg, w, device=local)
    if P:
        Wp, bp = synth.population(cfg, P)
        model.set_controllers(Wp, bp, pop_group=B // P)
    dev = torch.device("cuda", local)
    zc = torch.from_numpy(z0).to(dev)
    mc = torch.from_numpy(mask).to(dev)
    sh_dev = {} if shaping is None else {"rt0": torch.from_numpy(shaping[0]).to(dev),
                                         "mem0": torch.from_numpy(shaping[1]).to(dev)}
    if args.xfers:
        sh_dev["loc_mask"] = torch.from_numpy(loc_mask).to(dev)
    ep0 = rank * B
    out = {"z": torch.empty((T + 1, B, cfg["z_dim"]), device=dev),
           "actions": torch.empty((T, B), dtype=torch.int32, device=dev),
           "rewards": torch.empty((T, B), device=dev),
           "done": torch.empty((T, B), dtype=torch.uint8, device=dev)}
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)

    if P:  # a generation of a controller search: log-probs, values, returns and fitness too
        out["logp_seq"] = torch.empty((T, B), device=dev)
        out["value_seq"] = torch.empty((T, B), device=dev)
        ret = {"returns": torch.empty((T, B), device=dev)}

    def step():
        r = model.rollout(zc, T, mask=mc, episode_offset=ep0, want_final=False, out=out,
                          stream=stream, **sh_dev)
        n = model.last_launches
        if P:
            ret.update(model.returns(out["rewards"], out["done"], 0.99, bootstrap=out["value_seq"][T - 1],
                                     episode_offset=ep0, want_fitness=True, stream=stream))
            n += model.last_launches
        step.launches = n
        return r

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    path_name = model.last_path
    launches = step.launches
    if ws > 1:
        dist.barrier()
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    with ClockSampler(local) as clk:
        for i in range(args.steps):
            flush.fill_(float(i))
            ev[i][0].record(stream)
            step()
            ev[i][1].record(stream)
        torch.cuda.synchronize()
    if ws > 1:
        dist.barrier()
    times = [a.elapsed_time(b) for a, b in ev]  # ms, each one launch of the step
    # per-kernel durations: a second, identical timed pass with every kernel bracketed by CUDA
    # events on the launching stream (kept out of the pass above: the extra event records slow
    # calls made of many short launches)
    kt = kernel_timing_pass(model, step, flush, stream, args.steps)
    total_ms = max_over_ranks(sum(times), ws, dev)
    ms_per_step = total_ms / args.steps
    env_steps = B * T * ws
    live = None
    if cfg.get("done_terminates") or cfg.get("noop_terminates"):
        # episode b is live at step t unless it was done at an earlier step (then frozen);
        # every timed call computes the same trajectories, so the last one's done flags count
        d = out["done"].to(torch.int32)
        frozen = torch.zeros_like(d)
        frozen[1:] = (torch.cumsum(d, dim=0)[:-1] > 0).to(torch.int32)
        live_steps = int(sum_over_ranks(int((frozen == 0).sum().item()), ws, dev))
        live = {"live_env_steps": live_steps, "live_fraction": round(live_steps / env_steps, 4),
                "all_pairs_env_steps_per_s": round(env_steps / (ms_per_step / 1e3), 1)}
        env_steps = live_steps
    value = env_steps / (ms_per_step / 1e3)

    # e2e: the same call through the C ABI with pinned HOST buffers, copies timed.
    if args.no_e2e:
        e2e_value, h2d, d2h = None, 0, 0
    else:
        e2e_value, h2d, d2h = measure_e2e(model, z0, mask, T, ep0, args, flush, dev, ws, B, cfg,
                                          env_steps, shaping, loc_mask if args.xfers else None)

    # roofline of the dominant kernel: its algorithmic FLOPs per launch over its own
    # event-timed average launch duration inside the timed region
    peaks = load_peaks()
    timed = {k: v for k, v in kt.items() if k in KERNELS}
    dom = max(timed, key=lambda k: timed[k][0])
    dom_ms, dom_n = timed[dom]
    launch_ms = dom_ms / dom_n
    fl = kernel_flops(dom, cfg, B, T, dom_n)
    # the tensor family compacts the live episodes of a single controller before every step:
    # its GEMMs compute live rows only, so their algorithmic work is the live fraction's
    compacted = live is not None and path_name == "tensor" and not P
    if compacted:
        fl *= live["live_fraction"]
    achieved = fl / (launch_ms / 1e3) / 1e12
    unit = "TFLOP/s"
    if cfg["precision"] == "bf16" and dom in ("fused", "tc_ctrl", "tc_gates", "tc_heads"):
        bound = "tensor"
        # a call of the fused family is one short kernel (burst); the tensor family's kernels
        # run back to back inside a long call (sustained)
        burst = dom == "fused"
        peak = peaks["bf16_tflops"] if burst else peaks["bf16_tflops_sustained"]
        peak_source = f"{peaks['source']} bf16 {'burst' if burst else 'sustained'}"
    elif dom in ("tc_ctrl", "tc_gates", "tc_heads"):  # fp32 on the tensor cores: three bf16 passes
        bound, peak = "tensor", peaks["bf16_tflops_sustained"] / 3
        peak_source = f"{peaks['source']} bf16 sustained / 3 (fp32 products as three bf16 passes)"
    else:
        bound, peak = "alu", fp32_simt_peak_tflops()
        peak_source = "derived: 152 SM x 128 fp32 FMA x 2 FLOP x 2.07 GHz"
    kname, ksrc = KERNELS[dom]
    kernel_key = f"{kname}/{name}" + ("" if args.batch is None else f"@B{B}")
    traffic = ncu_traffic(kernel_key, kernel_source_sha(ksrc))
    all_ms = sum(v[0] for v in kt.values())
    roof = {"bound": bound, "achieved": round(achieved, 3), "peak": round(peak, 1), "unit": unit,
            "frac": round(achieved / peak, 5), "traffic": traffic, "peak_source": peak_source,
            "kernel": kernel_key, "launch_ms": round(launch_ms, 5), "launches": dom_n,
            "algorithmic_flops_per_launch": fl,
            "kernel_shares": {k: round(v[0] / all_ms, 4) for k, v in sorted(kt.items())}}

    line = {"metric": "dream env-steps/s (wm_rollout)", "value": round(value, 1),
            "unit": "env-steps/s", "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(ms_per_step, 4), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16" if cfg["precision"] == "bf16" else "f32",
            "data": "synthetic (seeded: weights N(0,0.05^2), z0 N(0,1), Bernoulli masks)",
            "config": {"workload": (name + ("+shaped_reward" if shaping is not None else "")
                                    + (f"+population{P}" if P else "")
                                    + (f"+hierarchical{args.xfers}" if args.xfers else ""))
                       if args.batch is None else f"{name} with B overridden",
                       "B": B, "T": T, "z": cfg["z_dim"], "A": cfg["a_dim"],
                       "H": cfg["h_dim"], "K": cfg["k_mix"],
                       "mask_density": synth.WORKLOADS[name]["mask_density"],
                       "precision": cfg["precision"], "kernel_path": path_name,
                       "reward": "Eq. 2 on predicted runtime / memory heads (alpha 0.8, beta 0.2, "
                                 "-100 invalid)" if shaping is not None else "linear reward head",
                       "action": "flat" if not args.xfers else
                       f"hierarchical: {args.xfers} xfers (incl. NO-OP) x {cfg['a_dim'] - args.xfers} "
                       "location slots (Sec. 3.1.3)",
                       "population": None if not P else
                       f"{P} controller candidates x {B // P} episodes; log-probs, value head, "
                       "discounted returns (gamma 0.99) and per-candidate fitness in the step",
                       "l2": "flushed between timed steps (512 MiB write)",
                       "parallelism": f"episodes sharded over {ws} GPU(s), no collective"},
            "e2e": None if e2e_value is None else
            {"value": round(e2e_value, 1), "unit": "env-steps/s",
             "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
            "gpu_launches": launches * args.steps,
            "roofline": roof, "clocks": clk.summary()}
    if live is not None:
        # value counts live pairs; the tensor family computes only those (compaction), the
        # other families also execute the frozen pairs
        live["frozen_pairs_executed"] = not compacted
        line["live_steps"] = live
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(name, args.cpu_episodes, shaped=shaping is not None)
    if rank == 0:
        print(json.dumps(line), flush=True)
    model.close()
    if ws > 1:
        dist.destroy_process_group()


def oracle_episodes(name: str, flop_budget: float) -> int:
    """Episodes whose whole rollout costs about flop_budget algorithmic FLOPs (bounded sample)."""
    w = synth.WORKLOADS[name]
    per = flops_per_env_step(synth.model_config(name)) * w["T"]
    return int(max(8, min(w["B"], flop_budget // per)))


def counted_steps(cfg: dict, done) -> int:
    """(episode, step) pairs a rollout counts: all of them, or the live ones when episodes
    can end (an episode is live at step t unless it was done at an earlier step)."""
    done = np.asarray(done)
    if not (cfg.get("done_terminates") or cfg.get("noop_terminates")):
        return int(done.size)
    ended = np.zeros_like(done, dtype=bool)
    ended[1:] = np.cumsum(done, axis=0)[:-1] > 0
    return int((~ended).sum())


def cpu_baseline(name: str, episodes: int | None, threads: int | None = None,
                 shaped: bool = False) -> dict:
    """The oracle on the host cores (all of them), plus a one-thread figure on a tenth of the
    sample (episodes are independent, so throughput per episode-step is comparable)."""
    import oracle

    cfg, w, z0, mask, B, T = synth.rollout_inputs(name)
    n = min(episodes or oracle_episodes(name, 2e11), B)
    threads = threads or os.cpu_count() or 1
    sh = {}
    if shaped:
        cfg["reward_mode"] = 1
        rt0, mem0 = synth.shaping_state(n)
        sh = {"rt0": rt0, "mem0": mem0}
    def timed(nn, nthreads, shs):
        """The sample's rollout, repeated until about 2 s have passed (a whole small workload
        takes milliseconds): (outputs, seconds per repetition, repetitions)."""
        reps, t0 = 0, time.perf_counter()
        while True:
            out = oracle.rollout(cfg, w, z0[:nn], mask[:, :nn], T, nthreads=nthreads, **shs)
            reps += 1
            dt = time.perf_counter() - t0
            if dt >= 2.0 or reps >= 1000:
                return out, dt / reps, reps

    o, dt, reps = timed(n, threads, sh)
    n1 = max(1, n // 10)
    o1, dt1, reps1 = timed(n1, 1, {k: v[:n1] for k, v in sh.items()})
    return {"value": round(counted_steps(cfg, o["done"]) / dt, 2), "unit": "env-steps/s",
            "cores": threads,
            "kind": "oracle", "sample": f"{n} of {B} episodes x {T} steps of {name}, "
                                        f"{threads} threads, {dt:.3g} s per repetition x {reps}",
            "value_1thread": round(counted_steps(cfg, o1["done"]) / dt1, 2),
            "sample_1thread": f"{n1} episodes x {T} steps, 1 thread, {dt1:.3g} s per repetition x {reps1}"}


def run_reference(args) -> None:
    ws, rank, _ = dist_env()
    if rank != 0:
        return
    import oracle

    name = args.workload
    if name == "nll":
        cfg = synth.model_config("nll", precision=args.precision or "bf16")
        w = synth.weights(cfg)
        zs, acts = nll_inputs(cfg)
        T, N = acts.shape
        n = max(8, min(N, args.ref_episodes or (N // 64 if args.train else N // 16)))
        threads = os.cpu_count() or 1
        fn = oracle.mdn_nll_grad if args.train else oracle.mdn_nll
        for _ in range(args.warmup):
            fn(cfg, w, zs[:, :n], acts[:, :n], nthreads=threads)
        times = []
        for _ in range(args.steps):
            t0 = time.perf_counter()
            fn(cfg, w, zs[:, :n], acts[:, :n], nthreads=threads)
            times.append(time.perf_counter() - t0)
        per = sum(times) / len(times)
        value = n * T / per
        metric = ("world-model training steps: scored (sequence, step) pairs/s (wm_mdn_nll_backward)"
                  if args.train else "teacher-forced scored steps/s (wm_mdn_nll)")
        line = {"impl": "reference", "metric": metric,
                "value": round(value, 2), "unit": "scored-steps/s", "n_gpus": ws, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": round(per * 1e3, 3), "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None,
                "dtype": "f64 (bf16 operand emulation)" if cfg["precision"] == "bf16" else "f64",
                "data": "synthetic (seeded: weights N(0,0.05^2), z ~ N(0,1), actions uniform)",
                "config": {"workload": f"nll_{cfg['precision']}" + ("_train" if args.train else ""), "N": N,
                           "T": T, "z": cfg["z_dim"], "A": cfg["a_dim"], "H": cfg["h_dim"], "K": cfg["k_mix"]},
                "cpu_baseline": {"value": round(value, 2), "unit": "scored-steps/s", "cores": threads,
                                 "kind": "oracle", "sample": f"{n} of {N} sequences x {T} steps, {threads} threads"},
                "e2e": {"value": round(value, 2), "unit": "scored-steps/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line), flush=True)
        return
    cfg, w, z0, mask, B, T = synth.rollout_inputs(name)
    n = min(args.ref_episodes or oracle_episodes(name, 2e10), B)
    threads = os.cpu_count() or 1
    for _ in range(args.warmup):
        oracle.rollout(cfg, w, z0[:n], mask[:, :n], T, nthreads=threads)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        o = oracle.rollout(cfg, w, z0[:n], mask[:, :n], T, nthreads=threads)
        times.append(time.perf_counter() - t0)
    per = sum(times) / len(times)
    value = counted_steps(cfg, o["done"]) / per
    sample = f"{n} of {B} episodes x {T} steps of {name} per step, {threads} threads"
    line = {"impl": "reference", "metric": "dream env-steps/s (wm_rollout)",
            "value": round(value, 2), "unit": "env-steps/s", "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(per * 1e3, 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None,
            "dtype": "f64 (bf16 operand emulation)" if cfg["precision"] == "bf16" else "f64",
            "data": "synthetic (seeded: weights N(0,0.05^2), z0 N(0,1), Bernoulli masks)",
            "config": {"workload": name, "B": B, "T": T, "z": cfg["z_dim"], "A": cfg["a_dim"],
                       "H": cfg["h_dim"], "K": cfg["k_mix"], "precision": cfg["precision"]},
            "cpu_baseline": {"value": round(value, 2), "unit": "env-steps/s", "cores": threads,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(value, 2), "unit": "env-steps/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="large_bf16", choices=list(synth.WORKLOADS),
                    help="a rollout workload, or nll (teacher-forced scoring)")
    ap.add_argument("--precision", choices=["fp32", "bf16"], default=None,
                    help="nll workload only: fp32 or bf16 path (default bf16)")
    ap.add_argument("--path", choices=["auto", "stepwise", "fused", "tensor"], default=None)
    ap.add_argument("--train", action="store_true",
                    help="nll workload: time the training step (loss and BPTT gradient)")
    ap.add_argument("--xfers", type=int, default=0,
                    help="hierarchical action: NX xfers (the last is the NO-OP) and A - NX "
                         "location slots (Sec. 3.1.3)")
    ap.add_argument("--population", type=int, default=0,
                    help="P controller candidates (B / P episodes each): each step is one "
                         "generation's evaluation (rollout with log-probs and values, returns, "
                         "fitness)")
    ap.add_argument("--reward", choices=["head", "shaped"], default="head",
                    help="rollout reward: the linear head, or Eq. 2 on the predicted runtime / "
                         "memory heads (Sec. 3.1.4)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true", help="skip the host-buffer leg (profiling runs)")
    ap.add_argument("--batch", type=int, default=None,
                    help="episodes per call instead of the workload's B (profiling runs only)")
    ap.add_argument("--cpu-episodes", type=int, default=None,
                    help="oracle sample size (default: about 2e11 FLOPs of the workload)")
    ap.add_argument("--ref-episodes", type=int, default=None,
                    help="oracle episodes per reference step (default: about 2e10 FLOPs)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        run_reference(args)
    elif args.workload == "nll" and args.train:
        run_train(args)
    elif args.workload == "nll":
        run_nll(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
