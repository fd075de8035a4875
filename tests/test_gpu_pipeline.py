"""End-to-end scoring slices on the GPU through the C-ABI, against the oracle:
  * the tiny workload (x [256 x 512], W 512x512, LoRA r=8, LM head 512 -> 4096,
    4 sequences x 64 tokens): compared in full;
  * the LM-head log-softmax/KL workload (h [2048 x 4096], LM head 4096 -> 32000 with a
    LoRA r=16 correction, lengths in [64, 512]): compared on seeded sampled rows."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2309_00754_gb300 import build as B
from paper_2309_00754_gb300 import hydra as H
from paper_2309_00754_gb300 import synth
from tests.helpers import (TOL_GAE, TOL_LINEAR, TOL_LOGP, assert_abs, assert_rel, dev_bf16,
                           dev_f32, dev_i32, f64, host_f64)

pytestmark = pytest.mark.gpu
BETA, GAMMA, LAM = 0.1, 1.0, 0.95


@pytest.fixture(scope="module", autouse=True)
def lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    B.build()
    H.load()
    H.device_error(clear=True)
    yield
    assert H.device_error(clear=True) == 0


def _ws(M, r):
    return torch.empty(max(1, H.lora_linear_workspace_size(M, r)), dtype=torch.uint8, device="cuda")


def test_tiny_scoring_pipeline_full():
    cfg = 1
    S, L, d, V, r, s = 4, 64, 512, 4096, 8, 2.0
    T = S * L
    g = lambda i: synth.tensor_seed(cfg, i)  # noqa: E731
    x = synth.normal_bf16(g(1), (T, d), 1.0)
    W = synth.normal_bf16(g(2), (d, d), 0.02)
    A = synth.normal_bf16(g(3), (r, d), 0.02)
    Bm = synth.normal_bf16(g(4), (d, r), 0.02)
    W_lm = synth.normal_bf16(g(5), (V, d), 0.02)
    ids = synth.randint(g(6), (T,), 0, V)
    values = synth.normal_f32(g(7), (S, L))
    score = synth.normal_f32(g(8), (S,))
    lengths = np.array([64, 50, 1, 64], dtype=np.int32)

    # GPU path: dual linear (shared input) -> LM head on both streams -> logp/KL -> GAE
    h_off = torch.empty(T, d, dtype=torch.bfloat16, device="cuda")
    h_on = torch.empty_like(h_off)
    H.hydra_lora_linear(dev_bf16(x), None, dev_bf16(W), dev_bf16(A), dev_bf16(Bm), s, h_off, h_on,
                        _ws(T, r))
    z_ref = torch.empty(T, V, device="cuda")
    z_act = torch.empty(T, V, device="cuda")
    H.hydra_lora_linear(h_off, h_on, dev_bf16(W_lm), None, None, s, z_ref, z_act, _ws(T, 0))
    la, lr, rw = (torch.empty(T, device="cuda") for _ in range(3))
    H.hydra_token_logprobs_kl(z_act, z_ref, dev_i32(ids), dev_i32(lengths), dev_f32(score), BETA,
                              S, L, la, lr, rw)
    adv = torch.empty(S, L, device="cuda")
    ret = torch.empty(S, L, device="cuda")
    H.ppo_gae(rw.view(S, L), dev_f32(values), dev_i32(lengths), GAMMA, LAM, adv, ret)

    # oracle
    o_off, o_on = O.dual_lora_linear(f64(x), f64(x), f64(W), f64(A), f64(Bm), s)
    assert_rel(host_f64(h_off), o_off, TOL_LINEAR, "h_off")
    assert_rel(host_f64(h_on), o_on, TOL_LINEAR, "h_on")
    oz_ref, oz_act = O.dual_lora_linear(o_off, o_on, f64(W_lm), None, None, s, out_bf16=False)
    assert_rel(host_f64(z_ref), oz_ref, TOL_LINEAR, "ref logits")
    assert_rel(host_f64(z_act), oz_act, TOL_LINEAR, "actor logits")
    ref = O.token_logprobs_kl(oz_act, oz_ref, ids, lengths, score, BETA, S, L)
    assert_abs(host_f64(la).reshape(S, L), ref["logp_actor"], TOL_LOGP, "logp_actor")
    assert_abs(host_f64(lr).reshape(S, L), ref["logp_ref"], TOL_LOGP, "logp_ref")
    assert_abs(host_f64(rw).reshape(S, L), ref["reward"], TOL_LOGP, "reward")
    # GAE given the GPU's own rewards: the scan's own tolerance
    a1, r1 = O.gae(host_f64(rw).reshape(S, L), values.astype(np.float64), lengths, GAMMA, LAM)
    assert_rel(host_f64(adv), a1, TOL_GAE, "advantages (same rewards)")
    assert_rel(host_f64(ret), r1, TOL_GAE, "returns (same rewards)")
    # end to end: reward error e propagates through sum_k (gamma lambda)^k <= 1/(1-gamma lambda)
    a_ref, r_ref = O.gae(ref["reward"], values.astype(np.float64), lengths, GAMMA, LAM)
    tol_e2e = TOL_LOGP / (1.0 - GAMMA * LAM) + TOL_GAE
    assert_rel(host_f64(adv), a_ref, tol_e2e, "advantages (end to end)")


def test_lm_head_logprobs_kl_sampled():
    cfg = 3
    S, L, d, V, r, s = 4, 512, 4096, 32000, 16, 2.0
    T = S * L
    g = lambda i: synth.tensor_seed(cfg, i)  # noqa: E731
    h = synth.normal_bf16(g(1), (T, d), 1.0)
    W_lm = synth.normal_bf16(g(2), (V, d), 0.02)
    A = synth.normal_bf16(g(3), (r, d), 0.02)
    Bm = synth.normal_bf16(g(4), (V, r), 0.02)
    ids = synth.randint(g(5), (T,), 0, V)
    lengths = synth.randint(g(6), (S,), 64, 513)
    score = synth.normal_f32(g(7), (S,))

    z_ref = torch.empty(T, V, device="cuda")
    z_act = torch.empty(T, V, device="cuda")
    H.hydra_lora_linear(dev_bf16(h), None, dev_bf16(W_lm), dev_bf16(A), dev_bf16(Bm), s, z_ref,
                        z_act, _ws(T, r))
    la, lr, rw = (torch.empty(T, device="cuda") for _ in range(3))
    H.hydra_token_logprobs_kl(z_act, z_ref, dev_i32(ids), dev_i32(lengths), dev_f32(score), BETA,
                              S, L, la, lr, rw)

    rows = set(int(v) for v in synth.randint(g(8), (48,), 0, T))
    for si in range(S):
        rows.update({si * L, si * L + int(lengths[si]) - 1, si * L + min(L - 1, int(lengths[si]))})
    rows = np.array(sorted(rows))
    oz_ref, oz_act = O.dual_lora_linear(f64(h[rows]), f64(h[rows]), f64(W_lm), f64(A), f64(Bm), s,
                                        out_bf16=False)
    assert_rel(host_f64(z_ref[rows]), oz_ref, TOL_LINEAR, "ref logits")
    assert_rel(host_f64(z_act[rows]), oz_act, TOL_LINEAR, "actor logits")
    ola, _ = O.log_softmax_gather(oz_act, ids[rows])
    olr, _ = O.log_softmax_gather(oz_ref, ids[rows])
    seq, t = rows // L, rows % L
    valid = t < lengths[seq]
    exp_la = np.where(valid, ola, 0.0)
    exp_lr = np.where(valid, olr, 0.0)
    exp_rw = np.where(valid, -BETA * (ola - olr), 0.0) + np.where(t == lengths[seq] - 1, score[seq], 0.0)
    assert_abs(host_f64(la[rows]), exp_la, TOL_LOGP, "logp_actor")
    assert_abs(host_f64(lr[rows]), exp_lr, TOL_LOGP, "logp_ref")
    assert_abs(host_f64(rw[rows]), exp_rw, TOL_LOGP, "reward")


# ------------------------------------------------------------------ fused LM head + log-softmax


def _fused_lm_head(h_off, h_on, W, A, Bm, s, ids, lengths, score, S, L):
    T = S * L
    V = W.shape[0]
    r = 0 if A is None else A.shape[0]
    ws = torch.empty(H.lm_head_logprobs_workspace_size(S, L, V, r), dtype=torch.uint8, device="cuda")
    out = [torch.full((T,), float("nan"), device="cuda") for _ in range(5)]
    H.hydra_lm_head_logprobs(h_off, h_on, W, A, Bm, s, ids, lengths, score, BETA, S, L, out[0],
                             out[1], out[2], ws, lse_actor=out[3], lse_ref=out[4])
    return out


@pytest.mark.parametrize("shared,V,r", [(True, 4096, 8), (False, 4096, 8), (False, 4104, 0),
                                        (True, 1000, 16)])
def test_fused_lm_head_logprobs(shared, V, r):
    """hydra_lm_head_logprobs (log-softmax partials in the GEMM epilogue) against the oracle's
    fp64 logits and log-softmax, and against the two-kernel GPU path; V = 4104 and 1000 leave
    a partial last 256-column tile."""
    S, L, d, s = 4, 64, 512, 2.0
    T = S * L
    g = lambda i: synth.tensor_seed(9, 100 * V + 10 * r + i)  # noqa: E731
    h0 = synth.normal_bf16(g(1), (T, d), 1.0)
    h1 = h0 if shared else synth.normal_bf16(g(2), (T, d), 1.0)
    W = synth.normal_bf16(g(3), (V, d), 0.02)
    A = synth.normal_bf16(g(4), (r, d), 0.02) if r else None
    Bm = synth.normal_bf16(g(5), (V, r), 0.02) if r else None
    ids = synth.randint(g(6), (T,), 0, V)
    lengths = np.array([64, 50, 1, 64], dtype=np.int32)
    score = synth.normal_f32(g(7), (S,))
    d_h0 = dev_bf16(h0)
    d_h1 = None if shared else dev_bf16(h1)
    dW, dA, dB = dev_bf16(W), dev_bf16(A) if r else None, dev_bf16(Bm) if r else None
    di, dl, dsc = dev_i32(ids), dev_i32(lengths), dev_f32(score)
    la, lr, rw, lsa, lsr = _fused_lm_head(d_h0, d_h1, dW, dA, dB, s, di, dl, dsc, S, L)

    oz_ref, oz_act = O.dual_lora_linear(f64(h0), f64(h1), f64(W), f64(A) if r else None,
                                        f64(Bm) if r else None, s, out_bf16=False)
    ref = O.token_logprobs_kl(oz_act, oz_ref, ids, lengths, score, BETA, S, L)
    assert_abs(host_f64(la).reshape(S, L), ref["logp_actor"], TOL_LOGP, "logp_actor")
    assert_abs(host_f64(lr).reshape(S, L), ref["logp_ref"], TOL_LOGP, "logp_ref")
    assert_abs(host_f64(rw).reshape(S, L), ref["reward"], TOL_LOGP, "reward")

    # the two-kernel path on the same inputs: equal up to the fp32 summation order
    z_ref = torch.empty(T, V, device="cuda")
    z_act = torch.empty(T, V, device="cuda")
    H.hydra_lora_linear(d_h0, d_h1, dW, dA, dB, s, z_ref, z_act, _ws(T, r))
    o = [torch.empty(T, device="cuda") for _ in range(5)]
    H.hydra_token_logprobs_kl(z_act, z_ref, di, dl, dsc, BETA, S, L, o[0], o[1], o[2], o[3], o[4])
    for got, want, name in zip((la, lr, rw, lsa, lsr), o, ("la", "lr", "rw", "lse_a", "lse_r")):
        assert_abs(host_f64(got), host_f64(want), 1e-4, f"fused vs two-kernel {name}")


def test_fused_lm_head_bad_token_id():
    S, L, d, V = 1, 16, 256, 1024
    h = dev_bf16(synth.normal_bf16(901, (S * L, d), 1.0))
    W = dev_bf16(synth.normal_bf16(902, (V, d), 0.02))
    ids_h = synth.randint(903, (S * L,), 0, V)
    ids_h[5] = V
    la, lr, rw, _, _ = _fused_lm_head(h, None, W, None, None, 1.0, dev_i32(ids_h), None, None, S, L)
    torch.cuda.synchronize()
    assert H.device_error(clear=True) == 0x201
    got = host_f64(la)
    assert np.isnan(got[5]) and np.isfinite(np.delete(got, 5)).all()


def test_fused_lm_head_c3_sampled():
    """The LM-head workload (h [2048 x 4096], 4096 -> 32000, LoRA r = 16, lengths in
    [64, 512]) through the fused path: all rows against the two-kernel path, sampled rows
    against the oracle."""
    cfg = 3
    S, L, d, V, r, s = 4, 512, 4096, 32000, 16, 2.0
    T = S * L
    g = lambda i: synth.tensor_seed(cfg, i)  # noqa: E731
    h = synth.normal_bf16(g(1), (T, d), 1.0)
    W_lm = synth.normal_bf16(g(2), (V, d), 0.02)
    A = synth.normal_bf16(g(3), (r, d), 0.02)
    Bm = synth.normal_bf16(g(4), (V, r), 0.02)
    ids = synth.randint(g(5), (T,), 0, V)
    lengths = synth.randint(g(6), (S,), 64, 513)
    score = synth.normal_f32(g(7), (S,))
    dh, dW, dA, dB = dev_bf16(h), dev_bf16(W_lm), dev_bf16(A), dev_bf16(Bm)
    di, dl, dsc = dev_i32(ids), dev_i32(lengths), dev_f32(score)
    la, lr, rw, _, _ = _fused_lm_head(dh, None, dW, dA, dB, s, di, dl, dsc, S, L)

    z_ref = torch.empty(T, V, device="cuda")
    z_act = torch.empty(T, V, device="cuda")
    H.hydra_lora_linear(dh, None, dW, dA, dB, s, z_ref, z_act, _ws(T, r))
    o = [torch.empty(T, device="cuda") for _ in range(3)]
    H.hydra_token_logprobs_kl(z_act, z_ref, di, dl, dsc, BETA, S, L, o[0], o[1], o[2])
    for got, want, name in zip((la, lr, rw), o, ("la", "lr", "rw")):
        assert_abs(host_f64(got), host_f64(want), 1e-4, f"fused vs two-kernel {name}")

    rows = np.array(sorted(set(int(v) for v in synth.randint(g(18), (16,), 0, T))))
    oz_ref, oz_act = O.dual_lora_linear(f64(h[rows]), f64(h[rows]), f64(W_lm), f64(A), f64(Bm), s,
                                        out_bf16=False)
    ola, _ = O.log_softmax_gather(oz_act, ids[rows])
    olr, _ = O.log_softmax_gather(oz_ref, ids[rows])
    seq, t = rows // L, rows % L
    valid = t < lengths[seq]
    assert_abs(host_f64(la[rows]), np.where(valid, ola, 0.0), TOL_LOGP, "logp_actor")
    assert_abs(host_f64(lr[rows]), np.where(valid, olr, 0.0), TOL_LOGP, "logp_ref")
