"""GPU parity: the CUDA path, called through the C-ABI, against the fp64 oracle on the same
seeded inputs. Small cases compare every element (several tiles, ragged tails); the
full-size workloads compare a seeded sample of rows, which the oracle computes one by
one (outputs are row-local, so the sample is an exact check of those rows)."""
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


@pytest.fixture(scope="module", autouse=True)
def lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    B.build()
    L = H.load()
    H.device_error(clear=True)
    yield L
    assert H.device_error(clear=True) == 0


def sample_rows(seed, M, n=64):
    rows = set(int(v) for v in synth.randint(seed, (n - 2,), 0, M))
    rows.update({0, M - 1})
    return np.array(sorted(rows))


# ------------------------------------------------------------------ GAE (a7)


@pytest.mark.parametrize("S,L,seed", [(4, 64, 1), (4, 512, 4), (64, 512, 5), (3, 37, 7),
                                      (5, 1000, 8), (2, 1, 9), (7, 33, 10), (9, 128, 11),
                                      (5, 384, 12), (3, 256, 13)])
def test_gae_parity(S, L, seed):
    r = synth.normal_f32(synth.tensor_seed(seed, 1), (S, L))
    v = synth.normal_f32(synth.tensor_seed(seed, 2), (S, L))
    lengths = synth.randint(synth.tensor_seed(seed, 3), (S,), 0, L + 1)
    lengths[0] = L
    if S > 2:
        lengths[1] = 0
        lengths[2] = min(1, L)
    adv = torch.empty(S, L, device="cuda")
    ret = torch.empty(S, L, device="cuda")
    H.ppo_gae(dev_f32(r), dev_f32(v), dev_i32(lengths), 1.0, 0.95, adv, ret)
    a_ref, r_ref = O.gae(r.astype(np.float64), v.astype(np.float64), lengths, 1.0, 0.95)
    assert_rel(host_f64(adv), a_ref, TOL_GAE, "advantages")
    assert_rel(host_f64(ret), r_ref, TOL_GAE, "returns")


def test_gae_no_lengths_and_discount():
    S, L = 3, 100
    r = synth.normal_f32(71, (S, L))
    v = synth.normal_f32(72, (S, L))
    adv = torch.empty(S, L, device="cuda")
    ret = torch.empty(S, L, device="cuda")
    H.ppo_gae(dev_f32(r), dev_f32(v), None, 0.99, 0.9, adv, ret)
    a_ref, r_ref = O.gae(r.astype(np.float64), v.astype(np.float64), None, 0.99, 0.9)
    assert_rel(host_f64(adv), a_ref, TOL_GAE, "advantages")
    assert_rel(host_f64(ret), r_ref, TOL_GAE, "returns")


def test_gae_large_batch_sampled():
    S, L = 65536, 512
    r = synth.normal_f32(81, (S, L))
    v = synth.normal_f32(82, (S, L))
    lengths = synth.randint(83, (S,), 64, 513)
    adv = torch.empty(S, L, device="cuda")
    ret = torch.empty(S, L, device="cuda")
    H.ppo_gae(dev_f32(r), dev_f32(v), dev_i32(lengths), 1.0, 0.95, adv, ret)
    rows = sample_rows(84, S)
    a_ref, r_ref = O.gae(r[rows].astype(np.float64), v[rows].astype(np.float64), lengths[rows], 1.0, 0.95)
    assert_rel(host_f64(adv[rows]), a_ref, TOL_GAE, "advantages")
    assert_rel(host_f64(ret[rows]), r_ref, TOL_GAE, "returns")


# ------------------------------------------------------------------ log-probs + KL (a4, a5)


def _logprobs_case(S, L, V, seed, dtype=torch.float32, ld=None, score=True, lengths=True):
    T = S * L
    ld = V if ld is None else ld
    za = synth.normal_f32(synth.tensor_seed(seed, 1), (T, ld), 1.3)
    zr = synth.normal_f32(synth.tensor_seed(seed, 2), (T, ld), 1.3)
    ids = synth.randint(synth.tensor_seed(seed, 3), (T,), 0, V)
    lens = synth.randint(synth.tensor_seed(seed, 4), (S,), 0, L + 1) if lengths else None
    if lens is not None:
        lens[0] = L
    sc = synth.normal_f32(synth.tensor_seed(seed, 5), (S,)) if score else None
    if dtype == torch.bfloat16:
        za_d = dev_bf16(synth.f32_to_bf16_bits(za))
        zr_d = dev_bf16(synth.f32_to_bf16_bits(zr))
        za64, zr64 = host_f64(za_d), host_f64(zr_d)
    else:
        za_d, zr_d = dev_f32(za), dev_f32(zr)
        za64, zr64 = za.astype(np.float64), zr.astype(np.float64)
    outs = [torch.full((T,), 7.0, device="cuda") for _ in range(5)]
    H.hydra_token_logprobs_kl(za_d[:, :V], zr_d[:, :V], dev_i32(ids),
                              None if lens is None else dev_i32(lens),
                              None if sc is None else dev_f32(sc), 0.1, S, L, *outs)
    ref = O.token_logprobs_kl(za64[:, :V], zr64[:, :V], ids, lens, sc, 0.1, S, L)
    names = ["logp_actor", "logp_ref", "reward", "lse_actor", "lse_ref"]
    for o, n in zip(outs, names):
        assert_abs(host_f64(o).reshape(S, L), ref[n], TOL_LOGP, n)


@pytest.mark.parametrize("S,L,V,seed", [(4, 64, 4096, 11), (3, 5, 1000, 12), (2, 7, 1, 13),
                                        (2, 9, 4099, 14), (1, 3, 3, 15)])
def test_logprobs_kl_parity(S, L, V, seed):
    _logprobs_case(S, L, V, seed)


def test_logprobs_kl_strided_bf16_and_no_score():
    _logprobs_case(3, 8, 4000, 16, ld=4096)
    _logprobs_case(3, 8, 4001, 17, ld=4003, score=False, lengths=False)
    _logprobs_case(2, 16, 32000, 18, dtype=torch.bfloat16)


def test_logprobs_kl_bad_id_flags_error():
    S, L, V = 1, 4, 64
    z = dev_f32(synth.normal_f32(19, (S * L, V)))
    ids = dev_i32(np.array([0, 64, 3, -1], dtype=np.int32))
    outs = [torch.zeros(S * L, device="cuda") for _ in range(3)]
    H.hydra_token_logprobs_kl(z, z, ids, None, None, 0.1, S, L, *outs)
    code = H.device_error(clear=True)
    assert code == 0x201
    la = outs[0].cpu().numpy()
    assert np.isfinite(la[0]) and np.isnan(la[1]) and np.isnan(la[3])


# ------------------------------------------------------------------ dual LoRA linear (a1-a3)


def _linear_problem(M, K, N, r, seed, std_x=1.0):
    x = synth.normal_bf16(synth.tensor_seed(seed, 1), (M, K), std_x)
    x2 = synth.normal_bf16(synth.tensor_seed(seed, 2), (M, K), std_x)
    W = synth.normal_bf16(synth.tensor_seed(seed, 3), (N, K), 0.02)
    A = synth.normal_bf16(synth.tensor_seed(seed, 4), (max(r, 1), K), 0.02)[:r]
    Bm = synth.normal_bf16(synth.tensor_seed(seed, 5), (N, max(r, 1)), 0.02)[:, :r]
    return x, x2, W, A, Bm


def _run_linear(x_off, x_on, W, A, Bm, s, out=torch.bfloat16, algo=0, want=(True, True)):
    M, K = x_off.shape
    N = W.shape[0]
    r = 0 if A is None else A.shape[0]
    y_off = torch.full((M, N), float("nan"), dtype=out, device="cuda") if want[0] else None
    y_on = torch.full((M, N), float("nan"), dtype=out, device="cuda") if want[1] else None
    ws = torch.empty(max(1, H.lora_linear_workspace_size(M, r)), dtype=torch.uint8, device="cuda")
    H.hydra_lora_linear(x_off, x_on, W, A, Bm, s, y_off, y_on, ws, algo=algo)
    return y_off, y_on


@pytest.mark.parametrize("M,K,N,r,shared,algo", [
    (256, 512, 512, 8, True, 1),      # config-1 first linear (CTA pairs)
    (256, 512, 512, 8, True, 3),      # same on single CTAs
    (300, 328, 520, 16, True, 1),     # ragged M, K (OOB k-block), N tail
    (300, 328, 520, 16, True, 3),
    (300, 328, 520, 16, False, 1),    # stacked streams
    (300, 328, 520, 16, False, 3),
    (129, 64, 256, 64, True, 1),
    (130, 1024, 768, 72, False, 1),   # two LoRA k-blocks
    (130, 1024, 768, 72, False, 3),
    (200, 512, 264, 128, True, 1),
    (700, 1024, 1280, 16, True, 1),   # several tiles per CTA pair (persistent loop)
    (700, 1024, 1280, 16, False, 1),
    (300, 256, 4264, 16, False, 1),   # CTA-pair tile widths 240, 208, 224 on GB300: stores of
    (300, 256, 3656, 16, False, 1),   # the columns past the last whole 64-column chunk
    (300, 256, 3960, 16, False, 1),
    (64, 256, 512, 0, True, 1),       # no LoRA
    (96, 256, 512, 0, False, 1),
    (400, 256, 512, 0, False, 1),
    (1, 4096, 4096, 16, True, 2),     # decode GEMV shapes
    (4, 4096, 1032, 16, True, 2),
    (8, 1024, 520, 8, False, 2),
    (16, 512, 512, 64, True, 2),
    (5, 1032, 1048, 16, False, 2),    # 10 token rows, K % 16 == 8 after two full chunks, N tail
    (3, 520, 72, 16, True, 0),
])
def test_lora_linear_parity(M, K, N, r, shared, algo):
    x, x2, W, A, Bm = _linear_problem(M, K, N, r, seed=M + K + N + r)
    xo = x if shared else x2
    y_off, y_on = _run_linear(dev_bf16(x), None if shared else dev_bf16(x2), dev_bf16(W),
                              dev_bf16(A) if r else None, dev_bf16(Bm) if r else None, 2.0,
                              algo=algo)
    ref_off, ref_on = O.dual_lora_linear(f64(x), f64(xo), f64(W), f64(A) if r else None,
                                         f64(Bm) if r else None, 2.0)
    assert_rel(host_f64(y_off), ref_off, TOL_LINEAR, "y_off")
    assert_rel(host_f64(y_on), ref_on, TOL_LINEAR, "y_on")


def test_lora_linear_fp32_out_and_single_outputs():
    M, K, N, r = 200, 256, 264, 16
    x, x2, W, A, Bm = _linear_problem(M, K, N, r, seed=21)
    d = [dev_bf16(t) for t in (x, x2, W, A, Bm)]
    ref_off, ref_on = O.dual_lora_linear(f64(x), f64(x2), f64(W), f64(A), f64(Bm), 2.0, out_bf16=False)
    y_off, y_on = _run_linear(d[0], d[1], d[2], d[3], d[4], 2.0, out=torch.float32)
    assert_rel(host_f64(y_off), ref_off, 1e-4, "y_off fp32")
    assert_rel(host_f64(y_on), ref_on, 1e-4, "y_on fp32")
    _, only_on = _run_linear(d[0], d[1], d[2], d[3], d[4], 2.0, out=torch.float32, want=(False, True))
    assert torch.equal(only_on, y_on)
    only_off, _ = _run_linear(d[0], d[0], d[2], d[3], d[4], 2.0, out=torch.float32, want=(True, False))
    ref_off_s, _ = O.dual_lora_linear(f64(x), f64(x), f64(W), f64(A), f64(Bm), 2.0, out_bf16=False)
    assert_rel(host_f64(only_off), ref_off_s, 1e-4, "y_off only")


@pytest.mark.parametrize("algo", [1, 2])
def test_lora_off_switch_is_bitwise(algo):
    # §3 Dynamic LoRA: with B = 0 (or s = 0) the LoRA-on output equals the LoRA-off output
    M = 16 if algo == 2 else 200
    K, N, r = 512, 264, 16
    x, _, W, A, _ = _linear_problem(M, K, N, r, seed=22)
    Bz = torch.zeros(N, r, dtype=torch.bfloat16, device="cuda")
    y_off, y_on = _run_linear(dev_bf16(x), None, dev_bf16(W), dev_bf16(A), Bz, 2.0, algo=algo)
    assert torch.equal(y_off, y_on)
    Bm = dev_bf16(synth.normal_bf16(23, (N, r), 0.02))
    y_off2, y_on2 = _run_linear(dev_bf16(x), None, dev_bf16(W), dev_bf16(A), Bm, 0.0, algo=algo)
    assert torch.equal(y_off2, y_on2) and torch.equal(y_off2, y_off)


@pytest.mark.parametrize("M,K,N", [
    (260, 384, 520),
    (2600, 4096, 1000),   # stacked input 43 MB: groups of 6 m-tiles over 11 (6 + 5)
    (2600, 11008, 512),   # stacked input 114 MB: groups of 4 over 11 (4 + 4 + 3); each
])                        # stream's own input 57 MB: groups of 4 in the separate calls
def test_stacked_equals_separate_calls_bitwise(M, K, N):
    """Stacked streams, separate calls and the grouped tile orders run the same per-tile
    arithmetic, so their outputs agree bit for bit."""
    r = 16
    x, x2, W, A, Bm = _linear_problem(M, K, N, r, seed=24)
    d = [dev_bf16(t) for t in (x, x2, W, A, Bm)]
    st_off, st_on = _run_linear(d[0], d[1], d[2], d[3], d[4], 2.0)
    sep_off, _ = _run_linear(d[0], None, d[2], d[3], d[4], 2.0)
    _, sep_on = _run_linear(d[1], None, d[2], d[3], d[4], 2.0)
    assert torch.equal(st_off, sep_off)
    assert torch.equal(st_on, sep_on)
    if M > 1000:  # the grouped orders against the oracle on sampled rows
        rows = sample_rows(M + N, M)
        ref_off, ref_on = O.dual_lora_linear(f64(x[rows]), f64(x2[rows]), f64(W), f64(A), f64(Bm), 2.0)
        assert_rel(host_f64(st_off[rows]), ref_off, TOL_LINEAR, "y_off")
        assert_rel(host_f64(st_on[rows]), ref_on, TOL_LINEAR, "y_on")


def test_gemv_and_tensor_core_kernel_agree():
    M, K, N, r = 16, 2048, 1024, 16
    x, _, W, A, Bm = _linear_problem(M, K, N, r, seed=25)
    d = [dev_bf16(t) for t in (x, W, A, Bm)]
    a = _run_linear(d[0], None, d[1], d[2], d[3], 2.0, algo=1)
    b = _run_linear(d[0], None, d[1], d[2], d[3], 2.0, algo=2)
    for u, v in zip(a, b):
        assert_rel(host_f64(u), host_f64(v), TOL_LINEAR, "gemv vs tcgen05")


@pytest.mark.parametrize("M,K,r", [
    (300, 4096, 64),     # streamed form, ragged last row block
    (3072, 4096, 32),    # q/v and gate/up of the full pass (clusters of 8 along K)
    (3072, 11008, 16),   # down projection of the full pass: 172 k-blocks, ragged split
    (2048, 4096, 16),    # LM head of the log-softmax workload
    (64, 1000, 8),       # one row block, K not a multiple of 64
    (65, 128, 24),       # two k-blocks only, rank 24 (three n-tiles of a 32-wide tile)
    (777, 4160, 136),    # three rank tiles of 64, the last partial
    (130, 72, 40),       # K just above one k-block
    (40, 4096, 16),      # below 64 rows: the register-fed form
    (16, 11008, 32),     # decode-sized
    (200, 48, 16),       # K below one k-block: the register-fed form
])
def test_lora_down_parity(M, K, r):
    x, _, _, A, _ = _linear_problem(M, K, 8, r, seed=26 + M + K + r)
    u = torch.full((M, r), float("nan"), dtype=torch.bfloat16, device="cuda")
    H.hydra_lora_down(dev_bf16(x), dev_bf16(A), 2.0, u)
    ref = O.lora_down(f64(x), f64(A), 2.0)
    assert_rel(host_f64(u), ref, TOL_LINEAR, "u")
    u2 = torch.empty_like(u)
    H.hydra_lora_down(dev_bf16(x), dev_bf16(A), 2.0, u2)
    assert torch.equal(u, u2), "lora_down is not deterministic"


# ------------------------------------------------------------------ full-size workloads


@pytest.mark.parametrize("K,N", [(4096, 4096), (4096, 11008), (11008, 4096)])
@pytest.mark.parametrize("r", [8, 16, 64])
def test_projection_sweep_sampled(K, N, r):
    """Llama-7B projection shapes at M = 2048 tokens (batch 4 x 512), shared input."""
    M = 2048
    x, _, W, A, Bm = _linear_problem(M, K, N, r, seed=2000 + K // 64 + N // 64 + r)
    y_off, y_on = _run_linear(dev_bf16(x), None, dev_bf16(W), dev_bf16(A), dev_bf16(Bm), 2.0)
    rows = sample_rows(2100 + r, M)
    ref_off, ref_on = O.dual_lora_linear(f64(x[rows]), f64(x[rows]), f64(W), f64(A), f64(Bm), 2.0)
    assert_rel(host_f64(y_off[rows]), ref_off, TOL_LINEAR, "y_off")
    assert_rel(host_f64(y_on[rows]), ref_on, TOL_LINEAR, "y_on")


@pytest.mark.parametrize("M", [1, 4, 8, 16])
def test_decode_gemv_sampled(M):
    """Decode-shaped inputs through the 4096 -> 32000 LM head, the 11008 -> 4096 down and the
    4096 -> 12288 q/k/v projection (whose 768 CTAs, up to 8 token rows, keep their partial
    tiles in the ring so that six fit on an SM and the grid is one wave)."""
    for K, N in ((4096, 32000), (11008, 4096), (4096, 12288)):
        x, _, W, A, Bm = _linear_problem(M, K, N, 16, seed=3000 + M + N)
        y_off, y_on = _run_linear(dev_bf16(x), None, dev_bf16(W), dev_bf16(A), dev_bf16(Bm), 2.0)
        ref_off, ref_on = O.dual_lora_linear(f64(x), f64(x), f64(W), f64(A), f64(Bm), 2.0)
        assert_rel(host_f64(y_off), ref_off, TOL_LINEAR, "y_off")
        assert_rel(host_f64(y_on), ref_on, TOL_LINEAR, "y_on")


# ------------------------------------------------------------------ fused epilogues


@pytest.mark.parametrize("shared", [True, False])
def test_swiglu_epilogue(shared):
    """Gate/up projection with the SwiGLU fused into the tcgen05 epilogue."""
    from paper_2309_00754_gb300 import llama
    M, K, F, r = 300, 512, 384, 16
    x, x2, _, _, _ = _linear_problem(M, K, 8, 8, seed=41)
    Wg = synth.normal_bf16(411, (F, K), 0.02)
    Wu = synth.normal_bf16(412, (F, K), 0.02)
    Bg = synth.normal_bf16(413, (F, r), 0.02)
    Bu = synth.normal_bf16(414, (F, r), 0.02)
    u = synth.normal_bf16(415, (M, 2 * r), 2.0)
    zg = np.zeros((F, r), np.uint16)
    Bcat_g = np.concatenate([Bg, zg], 1)
    Bcat_u = np.concatenate([zg, Bu], 1)
    W = llama.interleave_gate_up(Wg, Wu)
    B = llama.interleave_gate_up(Bcat_g, Bcat_u)
    xo = x if shared else x2
    y_off = torch.full((M, F), float("nan"), dtype=torch.bfloat16, device="cuda")
    y_on = torch.full((M, F), float("nan"), dtype=torch.bfloat16, device="cuda")
    H.hydra_dual_linear_ex(dev_bf16(x), None if shared else dev_bf16(x2), dev_bf16(W),
                           dev_bf16(u), dev_bf16(B), y_off, y_on, H.EPI_SWIGLU)
    uu = f64(u)
    g_off = O.round_bf16(f64(x) @ f64(Wg).T)
    u_off = O.round_bf16(f64(x) @ f64(Wu).T)
    g_on = O.round_bf16(f64(xo) @ f64(Wg).T + uu @ f64(Bcat_g).T)
    u_on = O.round_bf16(f64(xo) @ f64(Wu).T + uu @ f64(Bcat_u).T)
    assert_rel(host_f64(y_off), O.round_bf16(O.swiglu(g_off, u_off)), TOL_LINEAR, "swiglu off")
    assert_rel(host_f64(y_on), O.round_bf16(O.swiglu(g_on, u_on)), TOL_LINEAR, "swiglu on")


@pytest.mark.parametrize("shared,M,K,N", [(True, 260, 640, 520), (False, 260, 640, 520),
                                           (False, 300, 256, 4264), (False, 300, 256, 3656)])
def test_residual_epilogue(shared, M, K, N):
    """Projection added into an fp32 residual stream by the tcgen05 epilogue (the last two
    shapes take 240- and 208-column CTA-pair tiles on GB300: a 16-column tail per tile)."""
    r = 16
    x, x2, W, _, B = _linear_problem(M, K, N, r, seed=42)
    u = synth.normal_bf16(421, (M, r), 2.0)
    h0 = synth.normal_f32(422, (2, M, N), 3.0)
    h = dev_f32(h0)
    xo = x if shared else x2
    H.hydra_dual_linear_ex(dev_bf16(x), None if shared else dev_bf16(x2), dev_bf16(W),
                           dev_bf16(u), dev_bf16(B), h[0], h[1], H.EPI_RESIDUAL)
    y_off = O.round_bf16(f64(x) @ f64(W).T)
    y_on = O.round_bf16(f64(xo) @ f64(W).T + f64(u) @ f64(B).T)
    got = host_f64(h)
    assert_rel(got[0], h0[0].astype(np.float64) + y_off, TOL_LINEAR, "residual off")
    assert_rel(got[1], h0[1].astype(np.float64) + y_on, TOL_LINEAR, "residual on")


@pytest.mark.parametrize("N", [4264, 3656])
def test_fp32_output_tile_tails(N):
    """fp32 outputs with 240- / 208-column CTA-pair tiles (32-column store chunks + a 16-column
    tail per tile)."""
    M, K, r = 300, 256, 16
    x, x2, W, A, Bm = _linear_problem(M, K, N, r, seed=43 + N)
    y_off, y_on = _run_linear(dev_bf16(x), dev_bf16(x2), dev_bf16(W), dev_bf16(A), dev_bf16(Bm), 2.0,
                              out=torch.float32, algo=1)
    ref_off, ref_on = O.dual_lora_linear(f64(x), f64(x2), f64(W), f64(A), f64(Bm), 2.0, out_bf16=False)
    assert_rel(host_f64(y_off), ref_off, 1e-4, "y_off fp32")
    assert_rel(host_f64(y_on), ref_on, 1e-4, "y_on fp32")


@pytest.mark.parametrize("M,shared", [(300, False), (100, True), (700, False)])
def test_rope_epilogue(M, shared):
    """q/k/v projection with the rotary embedding fused into the tcgen05 epilogue: equal bit for
    bit to the projection followed by hydra_rope, and to the oracle's rotation of the
    bf16-rounded projection within the linear tolerance. M = 100 runs the single-CTA kernel."""
    H_, Dh, K, r, P, theta = 3, 128, 256, 16, 150, 10000.0
    d = H_ * Dh
    N = 3 * d
    x, x2, W, _, B = _linear_problem(M, K, N, r, seed=44 + M)
    u = synth.normal_bf16(441 + M, (M, r), 2.0)
    xs = [dev_bf16(t) for t in (x, x2, W, u, B)]
    x_on = None if shared else xs[1]
    ref = [torch.empty(M, N, dtype=torch.bfloat16, device="cuda") for _ in range(2)]
    H.hydra_dual_linear(xs[0], x_on, xs[2], xs[3], xs[4], ref[0], ref[1], algo=1)
    for t in ref:
        H.hydra_rope(t, d, Dh, P, theta)
    table = torch.empty(P, Dh // 2, 2, device="cuda")
    H.hydra_rope_table(P, Dh, theta, table)
    ang = np.arange(P)[:, None] * theta ** (-np.arange(Dh // 2) * 2.0 / Dh)[None, :]
    tab = host_f64(table)
    assert np.abs(tab[..., 0] - np.cos(ang)).max() < 1e-4 and np.abs(tab[..., 1] - np.sin(ang)).max() < 1e-4
    got = [torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda") for _ in range(2)]
    H.hydra_dual_linear_rope(xs[0], x_on, xs[2], xs[3], xs[4], got[0], got[1], P, 2 * d, Dh, table)
    assert torch.equal(got[0], ref[0]) and torch.equal(got[1], ref[1])
    xo = x if shared else x2
    pos = np.arange(M) % P
    for y_dev, inp, lora in ((got[0], x, False), (got[1], xo, True)):
        lin = f64(inp) @ f64(W).T + (f64(u) @ f64(B).T if lora else 0.0)
        lin = O.round_bf16(lin)
        want = lin.copy()
        for blk in range(2):
            want[:, blk * d:(blk + 1) * d] = O.round_bf16(
                O.rope(lin[:, blk * d:(blk + 1) * d].reshape(M, H_, Dh), pos, theta)).reshape(M, d)
        assert_rel(host_f64(y_dev), want, TOL_LINEAR, "rotary epilogue")


@pytest.mark.parametrize("M,K,N,r,out", [(300, 328, 520, 16, torch.bfloat16),
                                        (100, 256, 264, 8, torch.bfloat16),   # single-CTA tiles
                                        (700, 1024, 1280, 16, torch.bfloat16),  # several tiles per pair
                                        (260, 384, 4264, 16, torch.float32)])   # 240-wide pair tiles
def test_hydra_three_streams(M, K, N, r, out):
    """Hydra-PPO's off / actor / critic streams (two LoRA sets) through one W, against the
    oracle's dual-output linear of each LoRA set."""
    x, x2, W, A, Bm = _linear_problem(M, K, N, r, seed=61 + M)
    x3 = synth.normal_bf16(611 + M, (M, K), 1.0)
    A2 = synth.normal_bf16(612 + M, (r, K), 0.02)
    B2 = synth.normal_bf16(613 + M, (N, r), 0.02)
    ys = [torch.full((M, N), float("nan"), dtype=out, device="cuda") for _ in range(3)]
    ws = torch.empty(max(1, H.lora_linear_tri_workspace_size(M, r)), dtype=torch.uint8, device="cuda")
    H.hydra_lora_linear_tri(dev_bf16(x), dev_bf16(x2), dev_bf16(x3), dev_bf16(W), dev_bf16(A),
                            dev_bf16(Bm), dev_bf16(A2), dev_bf16(B2), 2.0, ys[0], ys[1], ys[2], ws)
    bf = out == torch.bfloat16
    tol = TOL_LINEAR if bf else 1e-4
    ref_off, ref_act = O.dual_lora_linear(f64(x), f64(x2), f64(W), f64(A), f64(Bm), 2.0, out_bf16=bf)
    _, ref_crit = O.dual_lora_linear(f64(x), f64(x3), f64(W), f64(A2), f64(B2), 2.0, out_bf16=bf)
    assert_rel(host_f64(ys[0]), ref_off, tol, "y_off")
    assert_rel(host_f64(ys[1]), ref_act, tol, "y_act")
    assert_rel(host_f64(ys[2]), ref_crit, tol, "y_crit")


def test_hydra_three_streams_reduce_to_two():
    """One LoRA set for actor and critic on one input (J-Hydra): the critic output equals the
    actor output and both equal the two-stream kernel's, bit for bit; an absent output is
    skipped."""
    M, K, N, r = 300, 512, 776, 16
    x, x2, W, A, Bm = _linear_problem(M, K, N, r, seed=71)
    d = [dev_bf16(t) for t in (x, x2, W, A, Bm)]
    ys = [torch.empty(M, N, dtype=torch.bfloat16, device="cuda") for _ in range(3)]
    ws = torch.empty(H.lora_linear_tri_workspace_size(M, r), dtype=torch.uint8, device="cuda")
    H.hydra_lora_linear_tri(d[0], d[1], d[1], d[2], d[3], d[4], d[3], d[4], 2.0, ys[0], ys[1], ys[2], ws)
    two = _run_linear(d[0], d[1], d[2], d[3], d[4], 2.0, algo=1)
    assert torch.equal(ys[2], ys[1]) and torch.equal(ys[1], two[1]) and torch.equal(ys[0], two[0])
    crit_only = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    H.hydra_lora_linear_tri(d[0], d[1], d[1], d[2], None, None, d[3], d[4], 2.0, None, None,
                            crit_only, ws)
    assert torch.equal(crit_only, ys[2])


def test_epilogue_argument_errors():
    x = torch.zeros(16, 64, dtype=torch.bfloat16, device="cuda")
    W = torch.zeros(200, 64, dtype=torch.bfloat16, device="cuda")
    y = torch.zeros(16, 100, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(H.HydraError) as e:  # SwiGLU needs N % 256 == 0
        H.hydra_dual_linear_ex(x, None, W, None, None, y, None, H.EPI_SWIGLU)
    assert e.value.status == 2
    with pytest.raises(H.HydraError) as e:
        H.hydra_dual_linear_ex(x, None, W, None, None, y, None, 7)
    assert e.value.status == 4
