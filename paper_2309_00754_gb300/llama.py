"""Llama-7B-shaped model weights in the layouts hydra_score_llama takes (include/hydra.h):
q/k/v fused into w_qkv [3d, d] with LoRA a_qv [2r, d] / b_qkv [3d, 2r] block-structured so
that q and v carry their own LoRA pair and k none; gate/up fused into w_gu [2F, d], their
rows interleaved in blocks of 128 (gate block j, then up block j) so that one 256-column
output tile holds matching gate and up features, with a_gu [2r, d] / b_gu [2F, 2r]; down
with its own rank-r pair. This module only arranges tensors; all arithmetic runs in
libhydra."""
from __future__ import annotations

import numpy as np
import torch

LLAMA7B = dict(n_layers=32, d_model=4096, n_heads=32, head_dim=128, ffn=11008, vocab=32000,
               prompt_len=256, response_len=512, lora_rank=16, lora_scale=2.0, rms_eps=1e-6,
               rope_theta=10000.0, beta=0.1, gamma=1.0, lam=0.95)

LAYER_KEYS = ("w_qkv", "a_qv", "b_qkv", "w_o", "w_gu", "a_gu", "b_gu", "w_down", "a_down",
              "b_down", "norm_attn", "norm_ffn")


def interleave_gate_up(gate, up, block=128):
    """Rows [g_0..g_127, u_0..u_127, g_128.., u_128.., ...] from gate [F, *] and up [F, *]
    (numpy or torch)."""
    F = gate.shape[0]
    assert F % block == 0 and up.shape[0] == F
    nb = F // block
    g = gate.reshape(nb, block, *gate.shape[1:])
    u = up.reshape(nb, block, *up.shape[1:])
    if isinstance(gate, np.ndarray):
        return np.stack([g, u], axis=1).reshape(2 * F, *gate.shape[1:])
    return torch.stack([g, u], dim=1).reshape(2 * F, *gate.shape[1:])


def deinterleave_gate_up(gu, block=128):
    """(gate, up) from rows interleaved by interleave_gate_up."""
    F = gu.shape[0] // 2
    nb = F // block
    x = gu.reshape(nb, 2, block, *gu.shape[1:])
    return x[:, 0].reshape(F, *gu.shape[1:]), x[:, 1].reshape(F, *gu.shape[1:])


def random_device_weights(cfg, seed, device, std=0.02):
    """Random-init weights drawn on the device in the fused layouts (benchmark data):
    matrices ~N(0, std^2), embedding and heads ~N(0, std^2), norm weights 1."""
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    d, F, V, r, n = cfg["d_model"], cfg["ffn"], cfg["vocab"], cfg["lora_rank"], cfg["n_layers"]
    bf = torch.bfloat16

    def rnd(*shape):
        return (std * torch.randn(*shape, device=device, generator=g)).to(bf)

    w = {k: [] for k in LAYER_KEYS}
    for _ in range(n):
        w["w_qkv"].append(rnd(3 * d, d))
        w["a_qv"].append(rnd(2 * r, d))
        b = torch.zeros(3 * d, 2 * r, dtype=bf, device=device)
        b[:d, :r] = rnd(d, r)
        b[2 * d:, r:] = rnd(d, r)
        w["b_qkv"].append(b)
        w["w_o"].append(rnd(d, d))
        w["w_gu"].append(rnd(2 * F, d))  # random rows: any interleave is equally random
        w["a_gu"].append(rnd(2 * r, d))
        bg = torch.zeros(F, 2 * r, dtype=bf, device=device)
        bu = torch.zeros(F, 2 * r, dtype=bf, device=device)
        bg[:, :r] = rnd(F, r)
        bu[:, r:] = rnd(F, r)
        w["b_gu"].append(interleave_gate_up(bg, bu))
        w["w_down"].append(rnd(d, F))
        w["a_down"].append(rnd(r, F))
        w["b_down"].append(rnd(d, r))
        w["norm_attn"].append(torch.ones(d, dtype=bf, device=device))
        w["norm_ffn"].append(torch.ones(d, dtype=bf, device=device))
    w["embed"] = rnd(V, d)
    w["final_norm"] = torch.ones(d, dtype=bf, device=device)
    w["lm_head"] = rnd(V, d)
    w["w_rm"] = rnd(d)
    return w


def random_device_lora(cfg, seed, device, std=0.02):
    """A second random LoRA set (the Hydra-PPO critic's) in the fused layouts of
    hydra_llama_lora, drawn on the device (benchmark data)."""
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    d, F, r, n = cfg["d_model"], cfg["ffn"], cfg["lora_rank"], cfg["n_layers"]
    bf = torch.bfloat16

    def rnd(*shape):
        return (std * torch.randn(*shape, device=device, generator=g)).to(bf)

    out = {k: [] for k in LORA_KEYS}
    for _ in range(n):
        out["a_qv"].append(rnd(2 * r, d))
        b = torch.zeros(3 * d, 2 * r, dtype=bf, device=device)
        b[:d, :r] = rnd(d, r)
        b[2 * d:, r:] = rnd(d, r)
        out["b_qkv"].append(b)
        out["a_gu"].append(rnd(2 * r, d))
        bg = torch.zeros(F, 2 * r, dtype=bf, device=device)
        bu = torch.zeros(F, 2 * r, dtype=bf, device=device)
        bg[:, :r] = rnd(F, r)
        bu[:, r:] = rnd(F, r)
        out["b_gu"].append(interleave_gate_up(bg, bu))
        out["a_down"].append(rnd(r, F))
        out["b_down"].append(rnd(d, r))
    return out


def fuse_separate(sep):
    """Fused numpy layouts (bf16 bit patterns, uint16) from separate per-projection arrays:
    sep has wq, wk, wv, wo [nl, d, d], wg, wu [nl, F, d], wd [nl, d, F], norm1, norm2
    [nl, d], embed [V, d], final_norm [d], lm_head [V, d], w_rm [d] and
    lora = {name: (A [nl, r, in], B [nl, out, r])} for name in wq, wv, wg, wu, wd."""
    nl = sep["wq"].shape[0]
    lo = sep["lora"]
    out = {k: [] for k in LAYER_KEYS}
    for l in range(nl):
        d = sep["wq"].shape[1]
        F = sep["wg"].shape[1]
        r = lo["wq"][0].shape[1]
        out["w_qkv"].append(np.concatenate([sep["wq"][l], sep["wk"][l], sep["wv"][l]], 0))
        out["a_qv"].append(np.concatenate([lo["wq"][0][l], lo["wv"][0][l]], 0))
        b = np.zeros((3 * d, 2 * r), dtype=np.uint16)
        b[:d, :r] = lo["wq"][1][l]
        b[2 * d:, r:] = lo["wv"][1][l]
        out["b_qkv"].append(b)
        out["w_o"].append(sep["wo"][l])
        out["w_gu"].append(interleave_gate_up(sep["wg"][l], sep["wu"][l]))
        out["a_gu"].append(np.concatenate([lo["wg"][0][l], lo["wu"][0][l]], 0))
        bg = np.zeros((F, 2 * r), dtype=np.uint16)
        bu = np.zeros((F, 2 * r), dtype=np.uint16)
        bg[:, :r] = lo["wg"][1][l]
        bu[:, r:] = lo["wu"][1][l]
        out["b_gu"].append(interleave_gate_up(bg, bu))
        out["w_down"].append(sep["wd"][l])
        out["a_down"].append(lo["wd"][0][l])
        out["b_down"].append(lo["wd"][1][l])
        out["norm_attn"].append(sep["norm1"][l])
        out["norm_ffn"].append(sep["norm2"][l])
    for k in ("embed", "final_norm", "lm_head", "w_rm"):
        out[k] = sep[k]
    return out


LORA_KEYS = ("a_qv", "b_qkv", "a_gu", "b_gu", "a_down", "b_down")


def fuse_lora(lora, d, F):
    """One LoRA set in the fused layouts of hydra_llama_lora (numpy bf16 bit patterns): lora =
    {name: (A [nl, r, in], B [nl, out, r])} for name in wq, wv, wg, wu, wd."""
    nl = lora["wq"][0].shape[0]
    r = lora["wq"][0].shape[1]
    out = {k: [] for k in LORA_KEYS}
    for l in range(nl):
        out["a_qv"].append(np.concatenate([lora["wq"][0][l], lora["wv"][0][l]], 0))
        b = np.zeros((3 * d, 2 * r), dtype=np.uint16)
        b[:d, :r] = lora["wq"][1][l]
        b[2 * d:, r:] = lora["wv"][1][l]
        out["b_qkv"].append(b)
        out["a_gu"].append(np.concatenate([lora["wg"][0][l], lora["wu"][0][l]], 0))
        bg = np.zeros((F, 2 * r), dtype=np.uint16)
        bu = np.zeros((F, 2 * r), dtype=np.uint16)
        bg[:, :r] = lora["wg"][1][l]
        bu[:, r:] = lora["wu"][1][l]
        out["b_gu"].append(interleave_gate_up(bg, bu))
        out["a_down"].append(lora["wd"][0][l])
        out["b_down"].append(lora["wd"][1][l])
    return out


def lora_to_device(fused, device):
    def dev(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(device)
    return {k: [dev(a) for a in fused[k]] for k in LORA_KEYS}


def to_device(fused, device):
    def dev(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(device)
    w = {k: [dev(a) for a in fused[k]] for k in LAYER_KEYS}
    for k in ("embed", "final_norm", "lm_head", "w_rm"):
        w[k] = dev(fused[k])
    return w


def alloc_outputs(S, L, device):
    o = {k: torch.empty(S, L, device=device) for k in
         ("logp_actor", "logp_ref", "reward", "values", "advantages", "returns")}
    o["score"] = torch.empty(S, device=device)
    return o
