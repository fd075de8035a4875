#!/usr/bin/env python
"""Throughput benchmark of the Hydra-PPO experience-scoring path on GB300.

One step = one pass of the scoring path over one batch of synthetic input, inputs resident
in HBM. Prints ONE JSON line (rank 0). Workloads:

  lm_head_scoring : final hidden states [4 x 512 x 4096] bf16 -> LoRA down (r=16) ->
                    dual-output LM head 4096 -> 32000 (fp32 logits, both streams, one pass
                    over W) -> sampled-token log-probs + KL reward (beta 0.1, score at the
                    last token, lengths U[64, 512]) -> GAE (gamma 1, lambda 0.95) with
                    per-token values ~ N(0, 1).

Metric: scored tokens/s = valid response tokens that received logp_actor, logp_ref, the
KL-penalised reward, the advantage and the return, per second.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Multi-GPU (torchrun): every rank scores its own batch (sequences are independent), there
is no data-path collective; value = all ranks' tokens / max-over-ranks time (weak scaling).
"""
from __future__ import annotations

import argparse
import json
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

METRIC = "scored tokens/s (actor+ref logprobs, KL, GAE) on 1 GB300; % of BF16/HBM roofline"
UNIT = "tokens/s"


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d["bf16_tflops_sustained"], "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


# ----------------------------------------------------------------------------- clocks


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(prefix="clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.15)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx.append(float(parts[2]))
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower().startswith("active"):
                        reasons.add(n)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": sorted(reasons),
                "samples": len(sm)}


# ----------------------------------------------------------------------------- workloads


class LmHeadScoring:
    """Final hidden states -> dual LM head -> log-probs + KL reward -> GAE."""

    name = "lm_head_scoring"
    S, L, d, V, r, s = 4, 512, 4096, 32000, 16, 2.0
    beta, gamma, lam = 0.1, 1.0, 0.95
    default_steps, default_warmup = 300, 10

    def __init__(self, device, seed=3):
        import torch
        from paper_2309_00754_gb300 import hydra as H
        from paper_2309_00754_gb300 import synth
        self.H = H
        self.dev = device
        S, L, d, V, r = self.S, self.L, self.d, self.V, self.r
        T = S * L
        self.T = T
        g = torch.Generator(device=device)
        g.manual_seed(seed)
        bf = torch.bfloat16
        self.h = torch.randn(T, d, device=device, generator=g).to(bf)
        self.W = (0.02 * torch.randn(V, d, device=device, generator=g)).to(bf)
        self.A = (0.02 * torch.randn(r, d, device=device, generator=g)).to(bf)
        self.B = (0.02 * torch.randn(V, r, device=device, generator=g)).to(bf)
        self.ids = torch.from_numpy(synth.randint(seed * 1000 + 5, (T,), 0, V)).to(device)
        self.lengths_np = synth.randint(seed * 1000 + 6, (S,), 64, 513)
        self.lengths = torch.from_numpy(self.lengths_np).to(device)
        self.score = torch.randn(S, device=device, generator=g)
        self.values = torch.randn(S, L, device=device, generator=g)
        self.u = torch.empty(T, r, dtype=bf, device=device)
        self.z_ref = torch.empty(T, V, device=device)
        self.z_act = torch.empty(T, V, device=device)
        self.la, self.lr, self.rw = (torch.empty(T, device=device) for _ in range(3))
        self.adv = torch.empty(S, L, device=device)
        self.ret = torch.empty(S, L, device=device)
        self.units = int(self.lengths_np.sum())
        self.launches_per_step = 4
        # algorithmic work of each kernel per launch
        self.gemm_flops = 2.0 * T * d * V + 2.0 * T * r * V
        valid_rows = self.units
        self.logp_bytes = valid_rows * V * 4 * 2 + T * (4 + 4 * 3) + S * 8
        self.gae_bytes = S * L * 16 + S * 4
        self.down_bytes = T * d * 2 + r * d * 2 + T * r * 2

    def step(self, ev=None):
        H = self.H
        if ev:
            ev["down"][0].record()
        H.hydra_lora_down(self.h, self.A, self.s, self.u)
        if ev:
            ev["down"][1].record()
            ev["gemm"][0].record()
        H.hydra_dual_linear(self.h, None, self.W, self.u, self.B, self.z_ref, self.z_act)
        if ev:
            ev["gemm"][1].record()
            ev["logp"][0].record()
        H.hydra_token_logprobs_kl(self.z_act, self.z_ref, self.ids, self.lengths, self.score,
                                  self.beta, self.S, self.L, self.la, self.lr, self.rw)
        if ev:
            ev["logp"][1].record()
            ev["gae"][0].record()
        H.ppo_gae(self.rw.view(self.S, self.L), self.values, self.lengths, self.gamma, self.lam,
                  self.adv, self.ret)
        if ev:
            ev["gae"][1].record()

    # end-to-end through the public API: per-step inputs come from pinned host memory and
    # the per-token results go back to pinned host memory
    def e2e_setup(self):
        import torch
        self.h_host = self.h.cpu().pin_memory()
        self.ids_host = self.ids.cpu().pin_memory()
        self.len_host = self.lengths.cpu().pin_memory()
        self.score_host = self.score.cpu().pin_memory()
        self.val_host = self.values.cpu().pin_memory()
        self.out_host = torch.empty(5, self.T, pin_memory=True)
        self.h2d = sum(t.numel() * t.element_size() for t in
                       (self.h_host, self.ids_host, self.len_host, self.score_host, self.val_host))
        self.d2h = self.out_host.numel() * 4

    def e2e_step(self):
        self.h.copy_(self.h_host, non_blocking=True)
        self.ids.copy_(self.ids_host, non_blocking=True)
        self.lengths.copy_(self.len_host, non_blocking=True)
        self.score.copy_(self.score_host, non_blocking=True)
        self.values.copy_(self.val_host, non_blocking=True)
        self.step()
        for i, t in enumerate((self.la, self.lr, self.rw, self.adv.view(-1), self.ret.view(-1))):
            self.out_host[i].copy_(t, non_blocking=True)

    def kernels(self, peaks, ms):
        """Per-kernel achieved throughput from mean event times (ms per launch)."""
        return {
            "dual_lora_gemm_tcgen05": {"ms": ms["gemm"], "TFLOP/s": self.gemm_flops / ms["gemm"] / 1e9},
            "logsoftmax_gather_kl": {"ms": ms["logp"], "GB/s": self.logp_bytes / ms["logp"] / 1e6},
            "gae_reverse_scan": {"ms": ms["gae"], "GB/s": self.gae_bytes / ms["gae"] / 1e6},
            "lora_down": {"ms": ms["down"], "GB/s": self.down_bytes / ms["down"] / 1e6},
        }

    def roofline(self, peaks, ms):
        achieved = self.gemm_flops / ms["gemm"] / 1e9
        peak = peaks["bf16_tflops_sustained"]
        return {"kernel": "dual_lora_gemm_tcgen05", "bound": "tensor", "achieved": achieved,
                "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak, "traffic": None,
                "peak_kind": f"bf16 dense, {peaks['source']} sustained"}

    def config(self):
        return {"workload": "lm_head_scoring: h[4x512x4096] -> dual LM head 4096->32000 (LoRA r=16, "
                            "s=2, fp32 logits) -> logp/KL (beta 0.1) -> GAE (gamma 1, lambda 0.95)",
                "batch": self.S, "response_len": self.L, "lengths": "U[64,512]",
                "scored_tokens_per_step": self.units, "l2": "inputs larger than L2 "
                "(W_lm 262 MB, logits 2 x 262 MB)"}

    # ---- CPU oracle on a bounded sample of the same workload
    def oracle_sample(self, n_rows):
        """Inputs for the oracle: the first n_rows token rows of sequence 0 (exact bf16 values)."""
        import oracle as O
        torch = __import__("torch")
        rows = np.arange(n_rows)

        def f64(t):
            return O.bf16_to_f64(t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16))
        return {"h": f64(self.h[rows]), "W": f64(self.W), "A": f64(self.A), "B": f64(self.B),
                "ids": self.ids[rows].cpu().numpy(), "score": self.score.cpu().numpy()[:1].astype(np.float64),
                "values": self.values[0:1, :n_rows].cpu().numpy().astype(np.float64), "n": n_rows}

    def oracle_run(self, smp):
        import oracle as O
        z_ref, z_act = O.dual_lora_linear(smp["h"], smp["h"], smp["W"], smp["A"], smp["B"], self.s,
                                          out_bf16=False)
        n = smp["n"]
        out = O.token_logprobs_kl(z_act, z_ref, smp["ids"], [n], smp["score"], self.beta, 1, n)
        O.gae(out["reward"], smp["values"], [n], self.gamma, self.lam)
        return n


WORKLOADS = {LmHeadScoring.name: LmHeadScoring}
DEFAULT_WORKLOAD = LmHeadScoring.name


# ----------------------------------------------------------------------------- helpers


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def max_over_ranks(value, world, device=None):
    """Max of a float over all ranks (identity when world == 1)."""
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world, device=None):
    if world > 1:
        import torch.distributed as dist
        if device is not None:
            dist.barrier(device_ids=[device.index])
        else:
            dist.barrier()


def time_oracle(wl, target_s=12.0):
    """Oracle throughput on a bounded sample (rank 0, host cores)."""
    probe = wl.oracle_sample(8)
    t0 = time.perf_counter()
    wl.oracle_run(probe)
    dt = time.perf_counter() - t0
    n = int(max(8, min(wl.L, 8 * target_s / max(dt, 1e-3))))
    smp = wl.oracle_sample(n)
    t0 = time.perf_counter()
    units = wl.oracle_run(smp)
    dt = time.perf_counter() - t0
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    return {"value": units / dt, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{units} token rows of sequence 0 through the fp64 oracle "
                      f"(LM head both streams, logp/KL, GAE) in {dt:.1f} s; BLAS threads = cores"}


# ----------------------------------------------------------------------------- arms


def run_reference(args, wl_cls):
    rank, world, local = dist_env()
    if rank != 0:
        return 0
    import torch
    if torch.cuda.is_available():
        torch.cuda.set_device(local)
    wl = wl_cls("cuda" if torch.cuda.is_available() else "cpu")
    smp = wl.oracle_sample(16)
    for _ in range(args.warmup):
        wl.oracle_run(smp)
    t0 = time.perf_counter()
    units = 0
    for _ in range(args.steps):
        units += wl.oracle_run(smp)
    dt = time.perf_counter() - t0
    value = units / dt
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": dt * 1e3 / max(1, args.steps),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "impl": "reference", "config": wl.config(),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": "16 token rows of sequence 0 per step through the fp64 oracle"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def run_ours(args, wl_cls):
    import torch
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    else:
        torch.cuda.set_device(0)
    device = torch.device("cuda", torch.cuda.current_device())
    import __graft_entry__
    __graft_entry__.build()
    from paper_2309_00754_gb300 import hydra as H
    H.device_error(clear=True)
    peaks = load_peaks()
    wl = wl_cls(device)
    steps = args.steps if args.steps is not None else wl.default_steps
    warmup = max(3, args.warmup if args.warmup is not None else wl.default_warmup)

    for _ in range(warmup):
        wl.step()
    torch.cuda.synchronize()
    if H.device_error(clear=True) != 0:
        raise RuntimeError("device error during warm-up")

    names = ("down", "gemm", "logp", "gae")
    evs = [{n: (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
            for n in names} for _ in range(steps)]
    clocks = ClockSampler(local)
    barrier(world, device)
    torch.cuda.synchronize()
    clocks.start()
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    start.record()
    for i in range(steps):
        wl.step(evs[i])
    end.record()
    torch.cuda.synchronize()
    barrier(world, device)
    clk = clocks.stop()
    ms_total = start.elapsed_time(end)
    ms_total_max = max_over_ranks(ms_total, world, device)
    per_kernel = {n: statistics.mean(e[n][0].elapsed_time(e[n][1]) for e in evs) for n in names}
    if H.device_error(clear=True) != 0:
        raise RuntimeError("device error during the timed steps")

    # end to end through the public API with host buffers
    wl.e2e_setup()
    for _ in range(2):
        wl.e2e_step()
    torch.cuda.synchronize()
    e2e_steps = max(3, min(steps, 50))
    barrier(world, device)
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(e2e_steps):
        wl.e2e_step()
    e1.record()
    torch.cuda.synchronize()
    barrier(world, device)
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), world, device)

    total_units = wl.units * steps * world
    value = total_units / (ms_total_max / 1e3)
    e2e_value = wl.units * e2e_steps * world / (e2e_ms / 1e3)
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": steps,
        "warmup": warmup, "ms_per_step": ms_total_max / steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": dict(wl.config(), parallelism=f"replicas{world}" if world > 1 else "single"),
        "roofline": wl.roofline(peaks, per_kernel),
        "kernels": wl.kernels(peaks, per_kernel),
        "clocks": clk,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": wl.h2d,
                "d2h_bytes_per_step": wl.d2h},
        "gpu_launches": wl.launches_per_step * steps,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = time_oracle(wl)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--warmup", type=int, default=None)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=sorted(WORKLOADS), default=DEFAULT_WORKLOAD)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args(argv)
    wl_cls = WORKLOADS[args.workload]
    if args.impl == "reference":
        if args.steps is None:
            args.steps = 20
        if args.warmup is None:
            args.warmup = 3
        return run_reference(args, wl_cls)
    return run_ours(args, wl_cls)


if __name__ == "__main__":
    sys.exit(main())
