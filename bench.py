#!/usr/bin/env python
"""Throughput benchmark of the Hydra-PPO experience-scoring path on GB300.

One step = one pass of the scoring path over one batch of synthetic input, inputs resident
in HBM. Prints ONE JSON line (rank 0). Workloads:

  hydra_scoring_llama7b (default) : the full J-Hydra scoring pass (hydra_score_llama) on a
                    random-init Llama-7B, batch 4 x (256 prompt + 512 response) tokens,
                    LoRA r=16 on q/v/gate/up/down, reward/value head 4096 -> 1.

  hydra_scoring_llama7b_400_400 : the same pass at the paper's sequence shape (Appendix B:
                    batch 4 x (400 prompt + 400 response)), for context.

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
                "bf16_tflops_sustained": d["bf16_tflops_sustained"], "source": "measured",
                "sustained_sm_mhz": d.get("clocks_under_load", {}).get("sm_mhz_median")}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback", "sustained_sm_mhz": None}


# nominal dense peaks of one GB300 (datasheet), reported beside the measured denominators
NOMINAL = {"TFLOP/s": 2250.0, "GB/s": 7900.0}


def annotate_roofline(roof, peaks, clk):
    """Secondary fractions beside the measured-peak one: against the nominal dense peak, and
    (tensor-bound, sustained peak) with both sides normalised by their median SM clock, since
    the measured sustained peak ran at a lower clock than the pass may."""
    if not roof or roof.get("achieved") is None:
        return roof
    nominal = NOMINAL.get(roof.get("unit"))
    if nominal:
        roof["frac_of_nominal"] = roof["achieved"] / nominal
        roof["nominal_peak"] = nominal
    mhz, peak_mhz = (clk or {}).get("sm_mhz"), peaks.get("sustained_sm_mhz")
    if (roof.get("bound") == "tensor" and "sustained" in roof.get("peak_kind", "") and mhz
            and peak_mhz):
        roof["frac_clock_normalised"] = (roof["achieved"] / mhz) / (roof["peak"] / peak_mhz)
        roof["clock_note"] = (f"pass median {mhz:.0f} MHz, measured sustained peak taken at "
                              f"median {peak_mhz:.0f} MHz")
    return roof


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
        # the timed region opens only once nvidia-smi has written its first sample: its
        # start-up (NVML initialisation) was seen to stall the GPU work submitted meanwhile
        t0 = time.time()
        while self.proc is not None and time.time() - t0 < 10.0:
            if self.proc.poll() is not None:
                break
            with open(self.path) as f:
                if f.readline():
                    break
            time.sleep(0.05)
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
    seed = 3
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
        # the fused LM head keeps per-tile log-softmax partials, never the logits
        self.ws = torch.empty(H.lm_head_logprobs_workspace_size(S, L, V, r), dtype=torch.uint8,
                              device=device)
        self.la, self.lr, self.rw = (torch.empty(T, device=device) for _ in range(3))
        self.adv = torch.empty(S, L, device=device)
        self.ret = torch.empty(S, L, device=device)
        self.units = int(self.lengths_np.sum())
        self.launches_per_step = 4  # lora_down, GEMM with log-softmax epilogue, combine, GAE
        self.event_names = ("gemm", "gae")  # CUDA-event pairs recorded by step()
        # algorithmic work per step: the LM head's flops (both heads, LoRA-up on the actor)
        self.gemm_flops = 2.0 * T * d * V + 2.0 * T * r * V
        self.gae_bytes = S * L * 16 + S * 4

    def step(self, ev=None):
        H = self.H
        if ev:
            ev["gemm"][0].record()
        H.hydra_lm_head_logprobs(self.h, None, self.W, self.A, self.B, self.s, self.ids,
                                 self.lengths, self.score, self.beta, self.S, self.L, self.la,
                                 self.lr, self.rw, self.ws)
        if ev:
            ev["gemm"][1].record()
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
            "lm_head_logprobs_fused": {"ms": ms["gemm"], "TFLOP/s": self.gemm_flops / ms["gemm"] / 1e9,
                                       "covers": "lora_down + tcgen05 LM head with log-softmax "
                                                 "epilogue + partial combine"},
            "gae_reverse_scan": {"ms": ms["gae"], "GB/s": self.gae_bytes / ms["gae"] / 1e6},
        }

    def roofline(self, peaks, ms):
        achieved = self.gemm_flops / ms["gemm"] / 1e9
        peak = peaks["bf16_tflops_sustained"]
        return {"kernel": "dual_lora_gemm_tcgen05 with the log-softmax epilogue (timed with its "
                          "lora_down and combine)", "bound": "tensor", "achieved": achieved,
                "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak, "traffic": None,
                "peak_kind": f"bf16 dense, {peaks['source']} sustained"}

    def config(self):
        return {"workload": "lm_head_scoring: h[4x512x4096] -> dual LM head 4096->32000 (LoRA r=16, "
                            "s=2) with the log-softmax reduced in the GEMM epilogue (no logits "
                            "stored) -> logp/KL (beta 0.1) -> GAE (gamma 1, lambda 0.95)",
                "batch": self.S, "response_len": self.L, "lengths": "U[64,512]",
                "scored_tokens_per_step": self.units, "l2": "inputs larger than L2 "
                "(W_lm 262 MB)"}

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


def oracle_layer_times(timer, smp, steps, warmup):
    """(t_head, [t_1 ...]): times of the oracle slice with no decoder layer (median of three)
    and with one decoder layer (`steps` samples). Both depths run once untimed first, so that
    neither carries the first call's thread start-up and page faults (a cold first call had
    made the head look slower than head + layer)."""
    timer(smp, 0)
    for _ in range(max(warmup, 1)):
        timer(smp, 1)
    t_head = statistics.median(timer(smp, 0) for _ in range(3))
    return t_head, [timer(smp, 1) for _ in range(steps)]


class HydraScoringLlama7B:
    """Full J-Hydra scoring pass on a random-init Llama-7B (32 layers, d 4096, 32 heads,
    SwiGLU 11008, vocab 32000, bf16), LoRA r=16 on q/v/gate/up/down (s = 2), reward head
    4096 -> 1 on the LoRA-off stream (values: same head on the LoRA-on stream); batch 4 x
    (256 prompt + 512 response) tokens -> actor/ref log-probs, reward, GAE."""

    name = "hydra_scoring_llama7b"
    seed = 4
    default_steps, default_warmup = 20, 3
    # DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum) per GEMM launch, averaged over
    # the 129 GEMM launches of one pass of this workload (batch 4, two streams): an ncu capture
    # of a three-layer pass (layer 0 with its shared q/k/v products, one full middle layer,
    # the last layer on its compact rows) and the LM head, the middle layer standing for the
    # 30 middle layers of the 32; no figure for other shapes or stream counts
    gemm_dram_bytes_per_launch = 490.4e6

    def __init__(self, device, seed=4, reference=False):
        import torch
        from paper_2309_00754_gb300 import llama, synth
        self.llama = llama
        self.cfg = dict(llama.LLAMA7B)
        c = self.cfg
        if getattr(self, "layers", None):  # fewer decoder layers: small profiling captures only
            c["n_layers"] = self.layers
        if getattr(self, "shape", None):  # (prompt, response) of a variant workload
            c["prompt_len"], c["response_len"] = self.shape
        self.S, self.P0, self.L = getattr(self, "batch", 4), c["prompt_len"], c["response_len"]
        self.beta, self.gamma, self.lam = c["beta"], c["gamma"], c["lam"]
        P = self.P0 + self.L
        self.weights = llama.random_device_weights(c, seed, device)
        self.ids = torch.from_numpy(synth.randint(seed * 1000 + 1, (self.S, P), 0, c["vocab"])).to(device)
        self.lengths = torch.full((self.S,), self.L, dtype=torch.int32, device=device)
        if not reference:  # the reference arm (fp64 oracle) never loads libhydra
            from paper_2309_00754_gb300 import hydra as H
            self.H = H
            self.ws = torch.empty(H.score_llama_workspace_size(c, self.S), dtype=torch.uint8,
                                  device=device)
            self.out = llama.alloc_outputs(self.S, self.L, device)
        self.units = int(self.S * self.L)
        T, SL = self.S * P, self.S * self.L
        d, F, V, r = c["d_model"], c["ffn"], c["vocab"], c["lora_rank"]
        nl = c["n_layers"]
        # algorithmic flops per pass of each projection class (both streams; LoRA-up on the
        # on stream only). Layer 0's q/k/v products serve both streams (equal inputs); the last
        # layer's o, gate/up and down run on the Tc rows the heads read (L + 1 per sequence).
        Tc = self.S * (self.L + 1) if self.L + 1 < P else T
        self.class_flops = {
            "gemm_qkv": (nl - 1) * (2 * (2 * T * d * 3 * d) + 2 * T * 2 * r * 3 * d)
                        + (2 * T * d * 3 * d + 2 * T * 2 * r * 3 * d),
            "gemm_o": (nl - 1) * 2 * (2 * T * d * d) + 2 * (2 * Tc * d * d),
            "gemm_gu": (nl - 1) * (2 * (2 * T * d * 2 * F) + 2 * T * 2 * r * 2 * F)
                       + (2 * (2 * Tc * d * 2 * F) + 2 * Tc * 2 * r * 2 * F),
            "gemm_down": (nl - 1) * (2 * (2 * T * F * d) + 2 * T * r * d)
                         + (2 * (2 * Tc * F * d) + 2 * Tc * r * d),
            "gemm_lmhead": 2 * (2 * SL * d * V),
        }
        self.gemm_flops = sum(self.class_flops.values())
        self.attn_flops = c["n_layers"] * 2 * self.S * c["n_heads"] * 2 * P * P * 128  # causal half
        # the log-probability class is the combine of the LM head's per-tile partials
        self.logp_bytes = SL * (2 * ((V + 255) // 256) * 8 + 2 * 4 + 4 + 12)
        self.launches_per_step = None

    def step(self, ev=None):
        self.H.hydra_score_llama(self.cfg, self.weights, self.ids, self.lengths, self.ws, self.out)

    def e2e_setup(self):
        import torch
        self.ids_host = self.ids.cpu().pin_memory()
        self.len_host = self.lengths.cpu().pin_memory()
        self.out_host = {k: torch.empty(v.shape, pin_memory=True) for k, v in self.out.items()}
        self.h2d = self.ids_host.numel() * 4 + self.len_host.numel() * 4
        self.d2h = sum(v.numel() * 4 for v in self.out_host.values())

    def e2e_step(self):
        self.ids.copy_(self.ids_host, non_blocking=True)
        self.lengths.copy_(self.len_host, non_blocking=True)
        self.step()
        for k, v in self.out.items():
            self.out_host[k].copy_(v, non_blocking=True)

    def kernels(self, peaks, prof):
        out = {}
        for k, (ms, n) in prof.items():
            if n:
                out[k] = {"ms_total": ms, "launches": n, "ms_per_launch": ms / n}
        for k, fl in self.class_flops.items():
            ms, n = prof[k]
            out[k]["TFLOP/s"] = fl * (n / self.launch_counts[k]) / ms / 1e9
        a = prof["attention"]
        out["attention"]["TFLOP/s"] = self.attn_flops * (a[1] / self.launch_counts["attention"]) / a[0] / 1e9
        lp = prof["logprobs"]
        out["logprobs"]["GB/s"] = self.logp_bytes * lp[1] / lp[0] / 1e6
        return out

    def traffic_per_launch(self):
        """The captured DRAM bytes per GEMM launch, for the exact workload they were taken on."""
        if (type(self) is HydraScoringLlama7B and self.S == 4 and not getattr(self, "shape", None)
                and self.cfg["n_layers"] == 32):
            return self.gemm_dram_bytes_per_launch
        return None

    def roofline(self, peaks, prof):
        ms = sum(prof[k][0] for k in self.class_flops)
        n = sum(prof[k][1] for k in self.class_flops)
        steps = n / sum(self.launch_counts[k] for k in self.class_flops)
        achieved = self.gemm_flops * steps / ms / 1e9
        peak = peaks["bf16_tflops_sustained"]
        return {"kernel": "dual_lora_gemm_tcgen05 (all projections + LM head of the pass)",
                "bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                "frac": achieved / peak, "traffic": self.traffic_per_launch(),
                "peak_kind": f"bf16 dense, {peaks['source']} sustained",
                "per_launch_flop": self.gemm_flops / sum(self.launch_counts[k] for k in self.class_flops),
                "per_launch_ms": ms / n,
                "timing": "CUDA events around every launch on the library's stream, over a second "
                          "run of the same steps right after the timed region",
                "profiled_ms_per_step": getattr(self, "profiled_ms_per_step", None)}

    def config(self):
        return {"workload": f"{self.name}: random-init Llama-7B ({self.cfg['n_layers']} layers, d 4096, 32 heads, "
                            "SwiGLU 11008, vocab 32000, bf16), LoRA r=16 s=2 on q/v/gate/up/down, reward/"
                            f"value head 4096->1; batch {self.S} x ({self.P0} prompt + {self.L} response); "
                            "logp/KL beta 0.1, GAE gamma 1 lambda 0.95",
                "batch": self.S, "prompt_len": self.P0, "response_len": self.L,
                "scored_tokens_per_step": self.units,
                "processed_tokens_per_step": 2 * self.S * (self.P0 + self.L),
                "l2": "inputs larger than L2 (13.5 GB of weights streamed per step)"}

    # ---- CPU oracle on a bounded slice of the same workload
    def oracle_sample(self, n_layers, prompt=32, resp=64):
        import oracle as O
        torch = __import__("torch")
        c = self.cfg
        d, F, r = c["d_model"], c["ffn"], c["lora_rank"]
        W = self.weights

        def f64(t):
            return O.bf16_to_f64(t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16))
        w = {"wq": [], "wk": [], "wv": [], "wo": [], "wg": [], "wu": [], "wd": [], "norm1": [],
             "norm2": [], "lora": {}}
        lo = {k: ([], []) for k in ("wq", "wv", "wg", "wu", "wd")}
        for l in range(n_layers):
            qkv = f64(W["w_qkv"][l])
            w["wq"].append(qkv[:d]); w["wk"].append(qkv[d:2 * d]); w["wv"].append(qkv[2 * d:])
            w["wo"].append(f64(W["w_o"][l]))
            g_, u_ = self.llama.deinterleave_gate_up(f64(W["w_gu"][l]))
            w["wg"].append(g_); w["wu"].append(u_)
            w["wd"].append(f64(W["w_down"][l]))
            w["norm1"].append(f64(W["norm_attn"][l])); w["norm2"].append(f64(W["norm_ffn"][l]))
            a, b = f64(W["a_qv"][l]), f64(W["b_qkv"][l])
            lo["wq"][0].append(a[:r]); lo["wq"][1].append(b[:d, :r])
            lo["wv"][0].append(a[r:]); lo["wv"][1].append(b[2 * d:, r:])
            a = f64(W["a_gu"][l])
            bg, bu = self.llama.deinterleave_gate_up(f64(W["b_gu"][l]))
            lo["wg"][0].append(a[:r]); lo["wg"][1].append(bg[:, :r])
            lo["wu"][0].append(a[r:]); lo["wu"][1].append(bu[:, r:])
            lo["wd"][0].append(f64(W["a_down"][l])); lo["wd"][1].append(f64(W["b_down"][l]))
        w = {k: (np.stack(v) if v else np.zeros((0,))) for k, v in w.items() if k != "lora"}
        w["lora"] = {k: (np.stack(a), np.stack(b)) for k, (a, b) in lo.items()}
        for k in ("embed", "final_norm", "lm_head", "w_rm"):
            w[k] = f64(W[k])
        ids = self.ids[0, self.P0 - prompt:self.P0 + resp].cpu().numpy()
        ocfg = {"d": d, "n_heads": c["n_heads"], "eps": c["rms_eps"], "lora_scale": c["lora_scale"],
                "rope_theta": c["rope_theta"], "n_layers": n_layers}
        return {"w": w, "ids": ids, "prompt": prompt, "resp": resp, "cfg": ocfg}

    def oracle_time(self, smp, n_layers):
        import oracle as O
        t0 = time.perf_counter()
        O.llama_score(smp["w"], smp["ids"], smp["prompt"], smp["cfg"], n_layers=n_layers,
                      beta=self.beta, gamma=self.gamma, lam=self.lam)
        return time.perf_counter() - t0

    def oracle_throughput(self, steps=1, single_thread=False, warmup=0):
        """(tokens/s, description): the slice's pass time is t(0 layers) + 32 (t(1) - t(0)); a
        quarter-size slice on one BLAS thread."""
        smp = self.oracle_sample(1, prompt=16, resp=32) if single_thread else self.oracle_sample(1)
        t_head, t1 = oracle_layer_times(self.oracle_time, smp, steps, warmup)
        self.oracle_timed = {"head_s": t_head, "sample_s": t1}
        n = self.cfg["n_layers"]
        t_pass = [t_head + n * max(t - t_head, 0.0) for t in t1]
        desc = (f"one sequence slice of {smp['prompt']} prompt + {smp['resp']} response tokens at full "
                f"width through the fp64 oracle: embed + heads {t_head:.2f} s, one decoder layer "
                f"{statistics.mean(t1) - t_head:.2f} s, pass time extrapolated to {n} layers")
        return smp["resp"] * len(t_pass) / sum(t_pass), desc


class HydraScoringLlama7BPaperShape(HydraScoringLlama7B):
    """The full J-Hydra scoring pass at the paper's sequence shape (Appendix B: batch 4,
    400-token prompts, 400-token completions), for context beside the 256 + 512 workload."""

    name = "hydra_scoring_llama7b_400_400"
    shape = (400, 400)


class HydraPPOScoringLlama7B(HydraScoringLlama7B):
    """Hydra-PPO scoring pass (Algorithm 2): the same model and batch as hydra_scoring_llama7b
    with a second, random LoRA set for the critic, so three streams (LoRA off, actor, critic)
    run through every layer; values come from the critic stream."""

    name = "hydra_ppo_scoring_llama7b"
    seed = 5

    def __init__(self, device, seed=5, reference=False):
        super().__init__(device, seed=seed, reference=reference)
        c = self.cfg
        self.critic = self.llama.random_device_lora(c, seed + 1000, device)
        if not reference:
            import torch
            self.ws = torch.empty(self.H.score_llama_hydra_workspace_size(c, self.S),
                                  dtype=torch.uint8, device=device)
        P = self.P0 + self.L
        T, SL = self.S * P, self.S * self.L
        d, F, V, r, nl = c["d_model"], c["ffn"], c["vocab"], c["lora_rank"], c["n_layers"]
        # three streams; the LoRA-up runs on the actor and critic streams; the last layer's o,
        # gate/up and down run on the Tc rows the heads read (L + 1 per sequence)
        Tc = self.S * (self.L + 1) if self.L + 1 < P else T
        self.class_flops = {
            "gemm_qkv": nl * (3 * (2 * T * d * 3 * d) + 2 * (2 * T * 2 * r * 3 * d)),
            "gemm_o": (nl - 1) * 3 * (2 * T * d * d) + 3 * (2 * Tc * d * d),
            "gemm_gu": (nl - 1) * (3 * (2 * T * d * 2 * F) + 2 * (2 * T * 2 * r * 2 * F))
                       + (3 * (2 * Tc * d * 2 * F) + 2 * (2 * Tc * 2 * r * 2 * F)),
            "gemm_down": (nl - 1) * (3 * (2 * T * F * d) + 2 * (2 * T * r * d))
                         + (3 * (2 * Tc * F * d) + 2 * (2 * Tc * r * d)),
            "gemm_lmhead": 2 * (2 * SL * d * V),
        }
        self.gemm_flops = sum(self.class_flops.values())
        self.attn_flops = nl * 3 * self.S * c["n_heads"] * 2 * P * P * 128  # causal half

    def step(self, ev=None):
        self.H.hydra_score_llama_hydra(self.cfg, self.weights, self.critic, self.ids, self.lengths,
                                       self.ws, self.out)

    def config(self):
        cfg = super().config()
        cfg["workload"] = ("hydra_ppo_scoring_llama7b: random-init Llama-7B (32 layers, d 4096, 32 "
                           "heads, SwiGLU 11008, vocab 32000, bf16), two LoRA sets r=16 s=2 (actor, "
                           "critic) on q/v/gate/up/down, reward/value head 4096->1; three streams; batch "
                           "4 x (256 prompt + 512 response); logp/KL beta 0.1, GAE gamma 1 lambda 0.95")
        cfg["processed_tokens_per_step"] = 3 * self.S * (self.P0 + self.L)
        return cfg

    def oracle_time(self, smp, n_layers):
        import oracle as O
        t0 = time.perf_counter()
        # the critic stream costs the same whichever set it carries: the actor's set stands in
        O.llama_score_hydra(smp["w"], smp["w"]["lora"], smp["ids"], smp["prompt"], smp["cfg"],
                            n_layers=n_layers, beta=self.beta, gamma=self.gamma, lam=self.lam)
        return time.perf_counter() - t0


class HydraGenerateLlama7B(HydraScoringLlama7B):
    """KV-cached generation (Algorithms 1 and 2: the actor generates each sequence for T
    steps, J-Hydra keeps the values) on the same random-init Llama-7B: 4 sequences of 256
    prompt tokens, 64 draws each from the actor's softmax (Gumbel-max, noise drawn on the
    device), the LoRA-off stream decoded beside the actor (reference log-probs of every
    draw), values and the final reward score. One step = one hydra_generate_llama call:
    prefill of both streams plus 64 decode steps of 8 rows (2 streams x 4 sequences)."""

    name = "hydra_generate_llama7b"
    seed = 6
    default_steps, default_warmup = 5, 3
    profiled = False
    event_names = ("gen",)
    metric = ("generated tokens/s (actor draws with logp_actor, logp_ref, values; both streams "
              "decoded) on 1 GB300; decode step vs HBM roofline")
    n_steps = 64
    batch = 4

    def __init__(self, device, seed=6, reference=False):
        super().__init__(device, seed=seed, reference=reference)
        import torch
        c = self.cfg
        S, V = self.S, c["vocab"]
        self.prompt = self.ids[:, :self.P0].contiguous()
        g = torch.Generator(device=device)
        g.manual_seed(seed * 1000 + 7)
        u = torch.rand(self.n_steps, S, V, device=device, generator=g).clamp_(1e-12, 1.0 - 1e-7)
        self.gumbel = -torch.log(-torch.log(u))
        del u
        if not reference:
            self.ws = torch.empty(self.H.generate_llama_workspace_size(c, S), dtype=torch.uint8,
                                  device=device)
            self.gen_out = {"tokens": torch.empty(S, self.n_steps, dtype=torch.int32, device=device),
                            "score": torch.empty(S, device=device)}
            for k in ("logp_actor", "logp_ref", "values"):
                self.gen_out[k] = torch.empty(S, self.n_steps, device=device)
        self.units = S * self.n_steps
        d, F, r, nl, H = c["d_model"], c["ffn"], c["lora_rank"], c["n_layers"], c["n_heads"]
        R = 2 * S
        # algorithmic bytes of one decode step: every weight once (bf16), the LoRA factors, the
        # cached keys and values up to the mean position, the new keys and values, the logits
        w_layer = (3 * d * d + d * d + 2 * F * d + d * F + 2 * d) * 2
        lora_layer = (2 * r * d + 3 * d * 2 * r + 2 * r * d + 2 * F * 2 * r + r * F + d * r) * 2
        mean_pos = self.P0 + self.n_steps / 2
        kv_layer = R * mean_pos * 2 * d * 2 + R * 2 * d * 2
        self.step_bytes = nl * (w_layer + lora_layer + kv_layer) + V * d * 2 + R * V * 4 * 2
        # launches of one call: prefill (rotary table, embed, 11 per layer, final norm, draw of
        # 3), each further draw (embed, 9 per layer, final norm, 3), the score pass (embed, 9
        # per layer, final norm, head)
        per_layer = 9
        decode = 1 + per_layer * nl + 1 + 3
        prefill = 2 + 11 * nl + 1 + 3
        self.launches_per_step = prefill + (self.n_steps - 1) * decode + (1 + per_layer * nl + 2)

    def _call(self, n_steps, out=None):
        o = out or self.gen_out
        if n_steps != self.n_steps:
            o = {k: (v[:, :n_steps].contiguous() if v.dim() == 2 else v) for k, v in o.items()}
        self.H.hydra_generate_llama(self.cfg, self.weights, self.prompt, n_steps, self.gumbel[:n_steps],
                                    self.ws, o)

    def step(self, ev=None):
        if ev is not None:
            ev["gen"][0].record()
        self._call(self.n_steps)
        if ev is not None:
            ev["gen"][1].record()

    def e2e_setup(self):
        import torch
        self.prompt_host = self.prompt.cpu().pin_memory()
        self.gumbel_host = self.gumbel.cpu().pin_memory()
        self.out_host = {k: torch.empty(v.shape, dtype=v.dtype, pin_memory=True)
                         for k, v in self.gen_out.items()}
        self.h2d = self.prompt_host.numel() * 4 + self.gumbel_host.numel() * 4
        self.d2h = sum(v.numel() * 4 for v in self.out_host.values())

    def e2e_step(self):
        self.prompt.copy_(self.prompt_host, non_blocking=True)
        self.gumbel.copy_(self.gumbel_host, non_blocking=True)
        self._call(self.n_steps)
        for k, v in self.gen_out.items():
            self.out_host[k].copy_(v, non_blocking=True)

    def _decode_step_ms(self, reps=3):
        """Decode step time from two call lengths: (T(n) - T(1)) / (n - 1), CUDA events."""
        import torch

        def timed(n):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for _ in range(reps):
                self._call(n)
            e1.record()
            torch.cuda.synchronize()
            return e0.elapsed_time(e1) / reps
        t1 = timed(1)
        tn = timed(self.n_steps)
        return (tn - t1) / (self.n_steps - 1), t1

    def kernels(self, peaks, ms):
        step_ms, t1 = self._decode_step_ms()
        self._step_ms = step_ms
        return {"generate_call": {"ms": ms["gen"]},
                "prefill_plus_first_draw": {"ms": t1},
                "decode_step": {"ms": step_ms, "GB/s": self.step_bytes / step_ms / 1e6,
                                "bytes": self.step_bytes}}

    def roofline(self, peaks, ms):
        step_ms = getattr(self, "_step_ms", None)
        if step_ms is None:
            step_ms, _ = self._decode_step_ms()
        achieved = self.step_bytes / step_ms / 1e6
        peak = peaks["hbm_gbs"]
        return {"kernel": "decode step (dual-output GEMV, or the tcgen05 GEMM above 16 rows, for every "
                          f"projection and the LM head; decode attention over the cache; fused norms): "
                          f"{2 * self.S} rows",
                "bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "traffic": None,
                "peak_kind": f"HBM copy, {peaks['source']}",
                "per_step_bytes": self.step_bytes, "per_step_ms": step_ms}

    def config(self):
        return {"workload": "hydra_generate_llama7b: random-init Llama-7B (32 layers, d 4096, 32 heads, "
                            f"SwiGLU 11008, vocab 32000, bf16), LoRA r=16 s=2 on q/v/gate/up/down; {self.S} "
                            f"sequences x 256 prompt tokens, {self.n_steps} Gumbel-max draws each; LoRA-off stream "
                            "decoded beside the actor; values and final score",
                "batch": self.S, "prompt_len": self.P0, "draws": self.n_steps,
                "generated_tokens_per_step": self.units,
                "l2": "inputs larger than L2 (13.5 GB of weights read per decode step)"}

    def oracle_time(self, smp, n_layers):
        import oracle as O
        t0 = time.perf_counter()
        O.llama_generate(smp["w"], smp["ids"][:smp["prompt"]], 2, smp["cfg"], n_layers=n_layers)
        return time.perf_counter() - t0

    def oracle_throughput(self, steps=1, single_thread=False, warmup=0):
        """(tokens/s, description): 2 draws after a 32-token prompt, per-draw time t(0 layers)
        + 32 (t(1) - t(0)), the oracle recomputing the whole prefix at each draw."""
        smp = self.oracle_sample(1)
        t_head, t1 = oracle_layer_times(self.oracle_time, smp, steps, warmup)
        self.oracle_timed = {"head_s": t_head, "sample_s": t1}
        n = self.cfg["n_layers"]
        t_gen = [t_head + n * max(t - t_head, 0.0) for t in t1]
        desc = (f"one sequence, {smp['prompt']} prompt tokens, 2 draws (plus the score pass) at full "
                f"width through the fp64 oracle, which recomputes the prefix at every draw: embed + "
                f"heads {t_head:.2f} s, one decoder layer {statistics.mean(t1) - t_head:.2f} s, time "
                f"extrapolated to {n} layers")
        return 2 * len(t_gen) / sum(t_gen), desc


class HydraPPOIterationLlama7B(HydraGenerateLlama7B):
    """One Hydra-PPO iteration's data path (Algorithm 2 without back-propagation) on the
    random-init Llama-7B: the actor generates 64 tokens after each of 4 prompts of 256
    (hydra_generate_llama, LoRA-off stream beside it), the drawn sequences go through the
    three-stream scoring pass with a second LoRA set for the critic (reference log-probs,
    reward, critic values, KL reward, GAE; hydra_score_llama_hydra), and the PPO losses and
    their gradients follow, with the generation's log-probs as the old policy and advantage
    whitening (hydra_ppo_loss). Both passes use the same weights, so the PPO ratio must be 1
    up to the two paths' numerics: the reported approx_kl and clip fraction check the
    KV-cached decode against the scoring pass at full size."""

    name = "hydra_ppo_iteration_llama7b"
    seed = 7
    default_steps, default_warmup = 3, 3
    event_names = ("gen", "score", "ppo")
    metric = ("experience tokens/s (Hydra-PPO iteration without back-propagation: generation, "
              "three-stream scoring, GAE, PPO losses) on 1 GB300; decode step vs HBM roofline")
    n_steps = 64

    def __init__(self, device, seed=7, reference=False):
        super().__init__(device, seed=seed, reference=reference)
        import torch
        c = self.cfg
        c["response_len"] = self.n_steps  # scoring covers exactly the drawn tokens
        S, n, P0 = self.S, self.n_steps, self.P0
        self.critic = self.llama.random_device_lora(c, seed + 1000, device)
        self.ids_buf = torch.empty(S, P0 + n, dtype=torch.int32, device=device)
        self.ids_buf[:, :P0].copy_(self.prompt)
        self.lengths = torch.full((S,), n, dtype=torch.int32, device=device)
        if not reference:
            H = self.H
            self.ws = torch.empty(H.generate_llama_workspace_size(c, S), dtype=torch.uint8,
                                  device=device)
            self.ws_score = torch.empty(H.score_llama_hydra_workspace_size(c, S),
                                        dtype=torch.uint8, device=device)
            self.score_out = self.llama.alloc_outputs(S, n, device)
            self.grad_logp = torch.empty(S, n, device=device)
            self.grad_values = torch.empty(S, n, device=device)
            self.stats = torch.zeros(7, dtype=torch.float64, device=device)
            self.ws_ppo = torch.empty(H.ppo_workspace_size(), dtype=torch.uint8, device=device)
        self.units = S * n

    def step(self, ev=None):
        def rec(k, i):
            if ev is not None:
                ev[k][i].record()
        rec("gen", 0)
        self._call(self.n_steps)
        rec("gen", 1)
        self.ids_buf[:, self.P0:].copy_(self.gen_out["tokens"])
        rec("score", 0)
        self.H.hydra_score_llama_hydra(self.cfg, self.weights, self.critic, self.ids_buf,
                                       self.lengths, self.ws_score, self.score_out)
        rec("score", 1)
        rec("ppo", 0)
        o = self.score_out
        self.H.hydra_ppo_loss(o["logp_actor"], self.gen_out["logp_actor"], o["advantages"],
                              o["returns"], o["values"], self.lengths, 0.2, True, self.grad_logp,
                              self.grad_values, self.stats, self.ws_ppo)
        rec("ppo", 1)

    def e2e_setup(self):
        import torch
        self.prompt_host = self.prompt.cpu().pin_memory()
        self.gumbel_host = self.gumbel.cpu().pin_memory()
        self.stats_host = torch.empty(7, dtype=torch.float64, pin_memory=True)
        self.tokens_host = torch.empty(self.S, self.n_steps, dtype=torch.int32, pin_memory=True)
        self.h2d = self.prompt_host.numel() * 4 + self.gumbel_host.numel() * 4
        self.d2h = self.stats_host.numel() * 8 + self.tokens_host.numel() * 4

    def e2e_step(self):
        self.prompt.copy_(self.prompt_host, non_blocking=True)
        self.ids_buf[:, :self.P0].copy_(self.prompt)
        self.gumbel.copy_(self.gumbel_host, non_blocking=True)
        self.step()
        self.stats_host.copy_(self.stats, non_blocking=True)
        self.tokens_host.copy_(self.gen_out["tokens"], non_blocking=True)

    def kernels(self, peaks, ms):
        import torch
        out = super().kernels(peaks, {"gen": ms["gen"]})
        out["scoring_hydra_ppo"] = {"ms": ms["score"]}
        out["ppo_loss"] = {"ms": ms["ppo"]}
        st = self.stats.cpu().tolist()
        out["ppo_stats_of_last_iteration"] = dict(zip(self.H.PPO_STATS, st))
        # decode path against the scoring pass on the same tokens and weights
        d = (self.score_out["logp_actor"] - self.gen_out["logp_actor"]).abs()
        dr = (self.score_out["logp_ref"] - self.gen_out["logp_ref"]).abs()
        out["decode_vs_scoring_max_abs_dlogp"] = {"actor": float(d.max()), "ref": float(dr.max())}
        # launches of the scoring pass, counted by the library's launch timing
        self.H.profile_enable(True)
        self.H.hydra_score_llama_hydra(self.cfg, self.weights, self.critic, self.ids_buf,
                                       self.lengths, self.ws_score, self.score_out)
        torch.cuda.synchronize()
        n_score = sum(n for _, n in self.H.profile_collect(reset=True).values())
        self.H.profile_enable(False)
        self.launches_per_step += n_score + 4  # + the PPO moments, coef, loss, finalize
        return out

    def config(self):
        return {"workload": "hydra_ppo_iteration_llama7b: random-init Llama-7B (32 layers, d 4096, 32 "
                            "heads, SwiGLU 11008, vocab 32000, bf16), actor and critic LoRA sets r=16 "
                            f"s=2; 4 sequences x 256 prompt tokens, {self.n_steps} Gumbel-max draws, "
                            "three-stream scoring (reference, actor, critic), KL reward beta 0.1, GAE "
                            "gamma 1 lambda 0.95, PPO losses clip 0.2 with whitening",
                "batch": self.S, "prompt_len": self.P0, "draws": self.n_steps,
                "experience_tokens_per_step": self.units,
                "l2": "inputs larger than L2 (13.5 GB of weights read per decode step)"}

    def oracle_time(self, smp, n_layers):
        import oracle as O
        t0 = time.perf_counter()
        gen = O.llama_generate(smp["w"], smp["ids"][:smp["prompt"]], 2, smp["cfg"], n_layers=n_layers)
        seq = np.concatenate([smp["ids"][:smp["prompt"]], gen["tokens"]])
        sc = O.llama_score_hydra(smp["w"], smp["w"]["lora"], seq, smp["prompt"], smp["cfg"],
                                 n_layers=n_layers, beta=self.beta, gamma=self.gamma, lam=self.lam)
        O.ppo_loss(sc["logp_actor"][None], gen["logp_actor"][None], sc["advantages"][None],
                   sc["returns"][None], sc["values"][None], [2], whiten=True)
        return time.perf_counter() - t0

    def oracle_throughput(self, steps=1, single_thread=False, warmup=0):
        smp = self.oracle_sample(1)
        t_head, t1 = oracle_layer_times(self.oracle_time, smp, steps, warmup)
        self.oracle_timed = {"head_s": t_head, "sample_s": t1}
        n = self.cfg["n_layers"]
        t_it = [t_head + n * max(t - t_head, 0.0) for t in t1]
        desc = (f"one sequence, {smp['prompt']} prompt tokens, 2 draws, three-stream scoring of the "
                f"result and the PPO losses at full width through the fp64 oracle: embed + heads "
                f"{t_head:.2f} s, one decoder layer {statistics.mean(t1) - t_head:.2f} s, time "
                f"extrapolated to {n} layers")
        return 2 * len(t_it) / sum(t_it), desc


class KernelSweep:
    """Per-kernel measurements of the rows the full pass does not exercise at their own
    shapes (one JSON line; value = the sweep's mean fraction of roofline):
      projection sweep: M = 2048 tokens through q/k/v/o (4096 -> 4096), gate/up
        (4096 -> 11008), down (11008 -> 4096), shared input, LoRA r in {8, 16, 64}, s = 2,
        both outputs -> TFLOP/s (the tensor-core dual-output kernel);
      decode: M in {1, 4, 8, 16} token rows through the distinct projection shapes
        (4096 -> 4096, 4096 -> 11008, 11008 -> 4096) and the 4096 -> 32000 LM head, r = 16,
        both outputs -> GB/s of W + x + u + y (the GEMV);
    Kernels are replayed back to back from CUDA graphs, weights rotated through copies
    larger than L2.
      GAE: 65536 sequences x 512 tokens -> GB/s;
      PPO losses (clipped surrogate, value loss, gradients, whitening): the same batch -> GB/s;
      causal attention: 8 sequences x 768 tokens x 32 heads of 128 -> TFLOP/s;
      log-probs/KL: 2048 rows x 32000 fp32 logits x 2 heads -> GB/s;
      LoRA down-projection: the full pass's and the LM head's shapes -> GB/s."""

    name = "kernel_sweep"
    seed = 5
    PROJ = (("q", 4096, 4096), ("k", 4096, 4096), ("v", 4096, 4096), ("o", 4096, 4096),
            ("gate", 4096, 11008), ("up", 4096, 11008), ("down", 11008, 4096))

    def __init__(self, device, seed=5, reference=False):
        self.device = device

    PARTS = ("projection_sweep", "decode", "decode_batch", "gae", "ppo_loss", "attention",
             "logprobs", "lora_down")

    def run(self, peaks, reps=20, parts=PARTS):
        import torch
        from paper_2309_00754_gb300 import hydra as H
        g = torch.Generator(device=self.device)
        g.manual_seed(self.seed)
        bf = torch.bfloat16
        dev = self.device

        def rnd(*shape, std=0.02):
            return (std * torch.randn(*shape, device=dev, generator=g)).to(bf)

        def graph_ms(launch, n, tag=None):
            """Mean time per launch of n back-to-back launches replayed from a CUDA graph
            (no host gaps between kernels). tag names an NVTX range around the measurement
            (for profiler filters: the first launch inside it runs outside any graph)."""
            if tag:
                torch.cuda.nvtx.range_push(tag)
            try:
                return _graph_ms(launch, n)
            finally:
                if tag:
                    torch.cuda.nvtx.range_pop()

        def _graph_ms(launch, n):
            launch(0)  # first call outside capture (one-time kernel attribute set-up)
            torch.cuda.synchronize()
            graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph):
                for i in range(n):
                    launch(i)
            graph.replay()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            graph.replay()
            e1.record()
            torch.cuda.synchronize()
            return e0.elapsed_time(e1) / n

        out = {k: {} for k in parts}
        # ---- projection sweep (c2): W rotates through 3 copies per shape so consecutive
        # launches do not find W in L2
        if "projection_sweep" in parts:
            M = 2048
            x = torch.randn(M, 11008, device=dev, generator=g).to(bf)
            fr = []
            for r in (8, 16, 64):
                for name, K, N in self.PROJ:
                    Ws = [rnd(N, K) for _ in range(3)]
                    B = rnd(N, r)
                    u = rnd(M, r, std=1.0)
                    xs = x[:, :K].contiguous()
                    y0 = torch.empty(M, N, dtype=bf, device=dev)
                    y1 = torch.empty(M, N, dtype=bf, device=dev)
                    ms = graph_ms(lambda i: H.hydra_dual_linear(xs, None, Ws[i % 3], u, B, y0, y1, algo=1), reps,
                                  tag=f"sweep:proj:{name}_r{r}")
                    tf = (2.0 * M * K * N + 2.0 * M * r * N) / ms / 1e9
                    out["projection_sweep"][f"{name}_r{r}"] = {"ms": ms, "TFLOP/s": tf}
                    fr.append(tf / peaks["bf16_tflops"])
                    del Ws
            sweep = out["projection_sweep"]
            sweep["mean_TFLOP/s"] = statistics.mean(v["TFLOP/s"] for v in list(sweep.values()))
            sweep["frac_of_measured_burst"] = statistics.mean(fr)
            sweep["frac_of_2.25PF"] = sweep["mean_TFLOP/s"] / 2250.0
        # ---- decode (c5): W rotates through enough copies that they exceed L2
        if "decode" in parts:
            shapes = list(self.PROJ[:1]) + list(self.PROJ[4:5]) + list(self.PROJ[6:]) + [("lm_head", 4096, 32000)]
            gb = []
            for n, K, N in shapes:
                ncopy = max(2, -(-300_000_000 // (N * K * 2)))  # > 2 x L2 of weights
                Wd = [rnd(N, K) for _ in range(ncopy)]
                Bd = rnd(N, 16)
                for Mt in (1, 4, 8, 16):
                    xd = torch.randn(Mt, K, device=dev, generator=g).to(bf)
                    ud = rnd(Mt, 16, std=1.0)
                    y0 = torch.empty(Mt, N, dtype=bf, device=dev)
                    y1 = torch.empty(Mt, N, dtype=bf, device=dev)
                    ms = graph_ms(lambda i: H.hydra_dual_linear(xd, None, Wd[i % ncopy], ud, Bd, y0, y1),
                                  max(reps, 2 * ncopy), tag=f"sweep:decode:{n}:M{Mt}")
                    byts = 2.0 * (N * K + 16 * (K + N) + Mt * K + 2 * Mt * N)
                    out["decode"].setdefault(f"M{Mt}", {})[n] = {"ms": ms, "GB/s": byts / ms / 1e6}
                    gb.append(byts / ms / 1e6)
                del Wd
            out["decode"]["frac_of_measured_hbm_mean"] = statistics.mean(gb) / peaks["hbm_gbs"]
        # ---- decode at 12 and 64 sequences: both streams' rows (24, 128) through the split-K
        # linear with the library's tile / cluster choice; W rotates through copies beyond L2
        if "decode_batch" in parts:
            shapes = (("qkv", 4096, 12288, 32), ("o", 4096, 4096, 0), ("gate_up", 4096, 22016, 32),
                      ("down", 11008, 4096, 16), ("lm_head", 4096, 32000, 0))
            gb = []
            for Mt in (24, 128):
                S = Mt // 2
                for n, K, N, r in shapes:
                    ncopy = max(2, -(-300_000_000 // (N * K * 2)))
                    Wd = [rnd(N, K) for _ in range(ncopy)]
                    Bd = rnd(N, r) if r else None
                    xd = torch.randn(Mt, K, device=dev, generator=g).to(bf)
                    ud = rnd(S, r, std=1.0) if r else None
                    yd = torch.empty(Mt, N, dtype=torch.float32 if n == "lm_head" else bf, device=dev)
                    ms = graph_ms(lambda i: H.hydra_skinny_linear(xd, Wd[i % ncopy], yd, u=ud, B=Bd,
                                                                  u_row0=S),
                                  max(reps, 2 * ncopy))
                    byts = 2.0 * (N * (K + r) + S * r + Mt * K) + yd.element_size() * Mt * N
                    out["decode_batch"].setdefault(f"M{Mt}", {})[n] = {"ms": ms, "GB/s": byts / ms / 1e6}
                    gb.append(byts / ms / 1e6)
                    del Wd
            out["decode_batch"]["frac_of_measured_hbm_mean"] = statistics.mean(gb) / peaks["hbm_gbs"]
            # launch cost: 128 rows x N 4096 with 128-column tiles, K of 1 to 64 k-blocks per
            # CTA, without a cluster and with 4 CTAs splitting K
            Wd = [rnd(4096, 4096) for _ in range(9)]
            xd = torch.randn(128, 4096, device=dev, generator=g).to(bf)
            yd = torch.empty(128, 4096, dtype=bf, device=dev)
            cost = {}
            for K in (64, 256, 1024, 4096):
                for ks in (1, 4):
                    if ks > K // 64:
                        continue
                    xk = xd[:, :K].contiguous()
                    Wk = [w[:, :K].contiguous() for w in Wd]
                    ms = graph_ms(lambda i: H.hydra_skinny_linear(xk, Wk[i % 9], yd, tile_n=128,
                                                                  split_k=ks), max(reps, 18))
                    cost[f"K{K}_split{ks}"] = {"us": ms * 1000.0}
                    del Wk
            out["decode_batch"]["launch_cost_N4096_M128_tile128"] = cost
            del Wd
        # ---- GAE at 65536 x 512
        if "gae" in parts or "ppo_loss" in parts:
            S, L = 65536, 512
            rw = torch.randn(S, L, device=dev, generator=g)
            vv = torch.randn(S, L, device=dev, generator=g)
            ln = torch.randint(64, 513, (S,), device=dev, generator=g, dtype=torch.int32)
            adv, ret = torch.empty_like(rw), torch.empty_like(rw)
            H.ppo_gae(rw, vv, ln, 1.0, 0.95, adv, ret)
            valid = float(ln.sum().item())
        if "gae" in parts:
            ms = graph_ms(lambda i: H.ppo_gae(rw, vv, ln, 1.0, 0.95, adv, ret), reps, tag="sweep:gae")
            byts = valid * 8 + S * L * 8 + S * 4  # read valid r, V; write all A, R
            out["gae"] = {"ms": ms, "GB/s": byts / ms / 1e6, "frac_of_measured_hbm": byts / ms / 1e6 / peaks["hbm_gbs"]}
        # ---- PPO losses at 65536 x 512, whitened: the moments pass reads the valid
        # advantages, the loss pass reads five fp32 inputs at valid tokens and writes both
        # gradient arrays in full
        if "ppo_loss" in parts:
            lo = -torch.randn(S, L, device=dev, generator=g).abs() * 2.0 - 0.05
            lnew = lo + 0.15 * torch.randn(S, L, device=dev, generator=g)
            gl, gv = torch.empty_like(lo), torch.empty_like(lo)
            st = torch.zeros(7, dtype=torch.float64, device=dev)
            ws = torch.empty(H.ppo_workspace_size(), dtype=torch.uint8, device=dev)
            ms = graph_ms(lambda i: H.hydra_ppo_loss(lnew, lo, rw, vv, ret, ln, 0.2, True, gl, gv, st, ws), reps)
            byts = valid * 24 + S * L * 8 + S * 8
            out["ppo_loss"] = {"ms": ms, "GB/s": byts / ms / 1e6, "frac_of_measured_hbm": byts / ms / 1e6 / peaks["hbm_gbs"],
                               "whiten": True}
            ms = graph_ms(lambda i: H.hydra_ppo_loss(lnew, lo, rw, vv, ret, ln, 0.2, False, gl, gv, st, ws), reps)
            byts = valid * 20 + S * L * 8 + S * 8
            out["ppo_loss"]["unwhitened"] = {"ms": ms, "GB/s": byts / ms / 1e6,
                                             "frac_of_measured_hbm": byts / ms / 1e6 / peaks["hbm_gbs"]}
            del lo, lnew, gl, gv
        if "gae" in parts or "ppo_loss" in parts:
            del rw, vv, adv, ret
        # ---- causal attention at the full pass's shape: 2 streams x 4 sequences x 768 tokens,
        # 32 heads of 128
        if "attention" in parts:
            nseq, Pq, Hh = 8, 768, 32
            qkv = torch.randn(nseq * Pq, 3 * Hh * 128, device=dev, generator=g).to(bf)
            att = torch.empty(nseq * Pq, Hh * 128, dtype=bf, device=dev)
            ms = graph_ms(lambda i: H.hydra_causal_attention(qkv, nseq, Pq, Hh, 128, att), reps,
                          tag="sweep:attention")
            fl = 4.0 * nseq * Hh * 128 * (Pq * (Pq + 1) / 2)  # q k^T and p v over the causal half
            out["attention"] = {"ms": ms, "TFLOP/s": fl / ms / 1e9}
            del qkv, att
        # ---- log-probs/KL at 2048 x 32000 x 2 heads, all rows valid
        if "logprobs" in parts:
            T, V = 2048, 32000
            za = torch.randn(T, V, device=dev, generator=g)
            zr = torch.randn(T, V, device=dev, generator=g)
            ids = torch.randint(0, V, (T,), device=dev, generator=g, dtype=torch.int32)
            o3 = [torch.empty(T, device=dev) for _ in range(3)]
            ms = graph_ms(lambda i: H.hydra_token_logprobs_kl(za, zr, ids, None, None, 0.1, 4, 512, *o3), reps,
                          tag="sweep:logprobs")
            byts = T * V * 4 * 2 + T * 16
            out["logprobs"] = {"ms": ms, "GB/s": byts / ms / 1e6, "frac_of_measured_hbm": byts / ms / 1e6 / peaks["hbm_gbs"]}
        # ---- LoRA down-projection at the full pass's shapes (3072 on-stream rows: q/v and
        # gate/up at K 4096 with 2 x 16 ranks, down at K 11008 with 16) and the LM-head
        # workload's (2048 x 4096, r 16); x rotates through copies beyond L2
        if "lora_down" in parts:
            for n, Mt, K, r in (("qv_gu", 3072, 4096, 32), ("down", 3072, 11008, 16),
                                ("lm_head", 2048, 4096, 16)):
                ncopy = max(2, -(-300_000_000 // (Mt * K * 2)))
                xs = [torch.randn(Mt, K, device=dev, generator=g).to(bf) for _ in range(ncopy)]
                A = rnd(r, K)
                u = torch.empty(Mt, r, dtype=bf, device=dev)
                ms = graph_ms(lambda i: H.hydra_lora_down(xs[i % ncopy], A, 2.0, u), max(reps, 2 * ncopy),
                              tag=f"sweep:lora_down:{n}")
                byts = 2.0 * (Mt * K + r * K + Mt * r)
                out["lora_down"][n] = {"ms": ms, "GB/s": byts / ms / 1e6,
                                       "frac_of_measured_hbm": byts / ms / 1e6 / peaks["hbm_gbs"]}
                del xs
        return out


WORKLOADS = {LmHeadScoring.name: LmHeadScoring, HydraScoringLlama7B.name: HydraScoringLlama7B,
             HydraScoringLlama7BPaperShape.name: HydraScoringLlama7BPaperShape,
             HydraPPOScoringLlama7B.name: HydraPPOScoringLlama7B,
             HydraGenerateLlama7B.name: HydraGenerateLlama7B,
             HydraPPOIterationLlama7B.name: HydraPPOIterationLlama7B,
             KernelSweep.name: KernelSweep}
DEFAULT_WORKLOAD = HydraScoringLlama7B.name


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


def aggregate(units_per_rank_step, steps, world, ms_max):
    """Whole-job throughput: every rank scores its own batch (weak scaling), so the job
    processes units_per_rank_step * steps * world units in the max-over-ranks time."""
    return units_per_rank_step * steps * world / (ms_max / 1e3)


def barrier(world, device=None):
    if world > 1:
        import torch.distributed as dist
        if device is not None:
            dist.barrier(device_ids=[device.index])
        else:
            dist.barrier()


_BLAS_THREAD_FNS = (("scipy_openblas_set_num_threads64_", "scipy_openblas_get_num_threads64_"),
                    ("scipy_openblas_set_num_threads", "scipy_openblas_get_num_threads"),
                    ("openblas_set_num_threads64_", "openblas_get_num_threads64_"),
                    ("openblas_set_num_threads", "openblas_get_num_threads"))


def blas_thread_control():
    """(get, set) for the thread count of the OpenBLAS that numpy loaded, or None: the library
    is found among this process's mapped files and driven through its exported setter."""
    import ctypes
    np.ones(2) @ np.ones(2)  # the BLAS is mapped once used
    try:
        with open("/proc/self/maps") as f:
            paths = {ln.split()[-1] for ln in f if len(ln.split()) >= 6 and "openblas" in ln.lower()}
    except OSError:
        return None
    for path in sorted(paths):
        try:
            lib = ctypes.CDLL(path)
        except OSError:
            continue
        for set_name, get_name in _BLAS_THREAD_FNS:
            if hasattr(lib, set_name) and hasattr(lib, get_name):
                setter, getter = getattr(lib, set_name), getattr(lib, get_name)
                setter.argtypes = [ctypes.c_int]
                getter.restype = ctypes.c_int
                return getter, setter
    return None


def single_thread_oracle(wl):
    """The oracle's throughput with BLAS on one thread (a smaller slice than the all-core leg)."""
    ctl = blas_thread_control()
    if ctl is None or not hasattr(wl, "oracle_throughput"):
        return None, "no OpenBLAS thread control found" if ctl is None else "not measured for this workload"
    get, set_ = ctl
    prev = get()
    try:
        set_(1)
        value, desc = wl.oracle_throughput(single_thread=True)
    finally:
        set_(prev)
    return value, desc + "; BLAS threads = 1"


def time_oracle(wl, target_s=12.0):
    """Oracle throughput on a bounded sample (rank 0, host cores), then on one thread."""
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    if hasattr(wl, "oracle_throughput"):
        value, desc = wl.oracle_throughput()
        st_value, st_desc = single_thread_oracle(wl)
        return {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                "sample": desc + "; BLAS threads = cores",
                "single_thread": {"value": st_value, "unit": UNIT, "cores": 1, "sample": st_desc}}
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
    if getattr(args, "gen_steps", None) and hasattr(wl_cls, "n_steps"):
        wl_cls.n_steps = args.gen_steps
    if getattr(args, "gen_batch", None) and hasattr(wl_cls, "n_steps"):
        wl_cls.batch = args.gen_batch
    rank, world, local = dist_env()
    if rank != 0:
        return 0
    import torch
    if torch.cuda.is_available():
        torch.cuda.set_device(local)
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    if hasattr(wl_cls, "oracle_throughput"):
        wl = wl_cls(dev, reference=True)
        value, desc = wl.oracle_throughput(steps=args.steps, warmup=args.warmup)
        timed = wl.oracle_timed
        # a step here is one timed oracle sample (the slice through embed, one decoder layer
        # and the heads); value is that sample extrapolated to the full pass, stated apart
        sample_ms = 1e3 * statistics.mean(timed["sample_s"])
        line = {"metric": getattr(wl, "metric", METRIC), "value": value, "unit": UNIT, "n_gpus": args.gpus,
                "steps": len(timed["sample_s"]), "warmup": args.warmup, "ms_per_step": sample_ms,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
                "data": "synthetic", "impl": "reference", "config": wl.config(),
                "extrapolated_from": {
                    "step": "one oracle sample: the slice through embed, one decoder layer and "
                            "the heads", "sample_ms": [1e3 * t for t in timed["sample_s"]],
                    "head_only_ms": 1e3 * timed["head_s"],
                    "full_pass_ms_extrapolated": 1e3 * wl.units / value,
                    "rule": "t(head) + n_layers x (t(sample) - t(head)), per full step of "
                            f"{wl.units} units"},
                "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                                 "sample": desc},
                "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line), flush=True)
        return 0
    wl = wl_cls(dev)
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


def run_sweep(args):
    import torch
    torch.cuda.set_device(0)
    import __graft_entry__
    __graft_entry__.build()
    peaks = load_peaks()
    clocks = ClockSampler(0)
    clocks.start()
    parts = tuple(args.parts.split(",")) if args.parts else KernelSweep.PARTS
    bad = [p for p in parts if p not in KernelSweep.PARTS]
    if bad:
        raise SystemExit(f"unknown --parts {bad}; choose from {','.join(KernelSweep.PARTS)}")
    res = KernelSweep(torch.device("cuda", 0)).run(peaks, parts=parts)
    clk = clocks.stop()
    line = {"metric": "per-kernel roofline fractions (projection sweep, decode GEMV, GAE, PPO losses, log-probs)",
            "value": res.get("projection_sweep", {}).get("frac_of_measured_burst"), "unit": "fraction",
            "workload": KernelSweep.name, "results": res, "clocks": clk, "peaks": peaks}
    print(json.dumps(line), flush=True)
    return 0


def run_ours(args, wl_cls):
    import torch
    if getattr(args, "gen_steps", None) and hasattr(wl_cls, "n_steps"):
        wl_cls.n_steps = args.gen_steps
    if getattr(args, "gen_batch", None) and hasattr(wl_cls, "n_steps"):
        wl_cls.batch = args.gen_batch
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
    wl = wl_cls(device, seed=wl_cls.seed + 100 * rank)  # every rank scores its own batch
    steps = args.steps if args.steps is not None else wl.default_steps
    warmup = max(3, args.warmup if args.warmup is not None else wl.default_warmup)

    for _ in range(warmup):
        wl.step()
    torch.cuda.synchronize()
    if H.device_error(clear=True) != 0:
        raise RuntimeError("device error during warm-up")

    driver = isinstance(wl, HydraScoringLlama7B) and getattr(wl, "profiled", True)
    names = getattr(wl, "event_names", ())
    evs = [None] * steps
    if driver:
        # launch counts of one pass (per-launch events on); the timed steps run without them
        H.profile_enable(True)
        wl.step()
        wl.launch_counts = {k: n for k, (_, n) in H.profile_collect(reset=True).items()}
        wl.launches_per_step = sum(wl.launch_counts.values())
        H.profile_enable(False)
        torch.cuda.synchronize()
    else:
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
    if driver:
        # per-kernel breakdown: the same K steps again, every launch bracketed by CUDA events
        # on the library's stream (kept out of the timed region above)
        H.profile_enable(True)
        torch.cuda.synchronize()
        p0 = torch.cuda.Event(enable_timing=True)
        p1 = torch.cuda.Event(enable_timing=True)
        p0.record()
        for i in range(steps):
            wl.step()
        p1.record()
        torch.cuda.synchronize()
        per_kernel = H.profile_collect(reset=True)
        H.profile_enable(False)
        wl.profiled_ms_per_step = p0.elapsed_time(p1) / steps
    else:
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

    value = aggregate(wl.units, steps, world, ms_total_max)
    e2e_value = aggregate(wl.units, e2e_steps, world, e2e_ms)
    metric = getattr(wl, "metric", METRIC)
    line = {
        "metric": metric, "value": value, "unit": UNIT, "n_gpus": world, "steps": steps,
        "warmup": warmup, "ms_per_step": ms_total_max / steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": dict(wl.config(), parallelism=f"replicas{world}" if world > 1 else "single"),
        "roofline": annotate_roofline(wl.roofline(peaks, per_kernel), peaks, clk),
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
    ap.add_argument("--layers", type=int, default=None,
                    help="scoring workloads only: decoder layers (default 32); fewer layers make "
                         "a small case for multi-pass profiler captures, never a bench value")
    ap.add_argument("--gen-steps", type=int, default=None,
                    help="generation workloads only: draws per call (default 64)")
    ap.add_argument("--gen-batch", type=int, default=None,
                    help="generation workloads only: sequences per call (default 4, at most 64)")
    ap.add_argument("--parts", default=None,
                    help="kernel_sweep only: comma-separated subset of " + ",".join(KernelSweep.PARTS))
    args = ap.parse_args(argv)
    wl_cls = WORKLOADS[args.workload]
    if args.layers is not None:
        if not issubclass(wl_cls, HydraScoringLlama7B):
            raise SystemExit("--layers applies to the scoring workloads only")
        wl_cls.layers = args.layers
    if wl_cls is KernelSweep:
        return run_sweep(args)
    if args.impl == "reference":
        if args.steps is None:
            args.steps = 3 if args.workload == HydraScoringLlama7B.name else 20
        if args.warmup is None:
            args.warmup = 3
        return run_reference(args, wl_cls)
    return run_ours(args, wl_cls)


if __name__ == "__main__":
    sys.exit(main())
