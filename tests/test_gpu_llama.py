"""GPU parity of the Llama decoder pieces and of the full J-Hydra scoring pass
(hydra_score_llama) against the fp64 oracle, through the C-ABI."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2309_00754_gb300 import build as Bld
from paper_2309_00754_gb300 import hydra as H
from paper_2309_00754_gb300 import llama, synth
from tests.helpers import (TOL_GAE, TOL_LINEAR, TOL_LOGP, assert_abs, assert_rel, dev_bf16,
                           dev_f32, dev_i32, f64, host_f64, max_abs_err)

pytestmark = pytest.mark.gpu
ONE_BF16 = np.uint16(0x3F80)


@pytest.fixture(scope="module", autouse=True)
def lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    Bld.build()
    H.load()
    H.device_error(clear=True)
    yield
    assert H.device_error(clear=True) == 0


# ------------------------------------------------------------------ pieces


def test_embed_two_copies_exact():
    V, d, T = 300, 256, 77
    table = synth.normal_bf16(501, (V, d), 0.02)
    ids = synth.randint(502, (T,), 0, V)
    h = torch.full((2 * T, d), float("nan"), device="cuda")
    H.hydra_embed(dev_bf16(table), dev_i32(ids), 2, h)
    ref = f64(table)[ids]
    got = host_f64(h)
    assert np.array_equal(got[:T], ref) and np.array_equal(got[T:], ref)


def test_rmsnorm_with_row_gather():
    d, S, P, L, p0 = 512, 3, 40, 25, 9
    x = synth.normal_f32(511, (2 * S * P, d), 1.5)
    w = synth.normal_bf16(512, (d,), 1.0)
    y = torch.empty(2 * S * L, d, dtype=torch.bfloat16, device="cuda")
    H.hydra_rmsnorm(dev_f32(x), dev_bf16(w), 1e-6, y, g_out=L, g_in=P, off=p0 - 1)
    rows = np.array([(i // L) * P + p0 - 1 + i % L for i in range(2 * S * L)])
    ref = O.round_bf16(O.rmsnorm(x[rows].astype(np.float64), f64(w), 1e-6))
    assert_rel(host_f64(y), ref, TOL_LINEAR, "rmsnorm")


def test_rope_q_k_rotated_v_untouched():
    H_, Dh, S, P = 3, 128, 2, 70
    d = H_ * Dh
    qkv_bits = synth.normal_bf16(521, (S * P, 3 * d), 1.0)
    qkv = dev_bf16(qkv_bits)
    H.hydra_rope(qkv, d, Dh, P, 10000.0)
    got = host_f64(qkv)
    x = f64(qkv_bits)
    pos = np.arange(S * P) % P
    for blk in range(2):
        ref = O.round_bf16(O.rope(x[:, blk * d:(blk + 1) * d].reshape(-1, H_, Dh), pos, 10000.0))
        assert_rel(got[:, blk * d:(blk + 1) * d], ref.reshape(-1, d), TOL_LINEAR, f"rope block {blk}")
    assert np.array_equal(got[:, 2 * d:], x[:, 2 * d:])


@pytest.mark.parametrize("nseq,P,H_,q_std", [(3, 100, 2, 1.0), (1, 768, 1, 1.0), (2, 64, 1, 1.0),
                                             (1, 1, 2, 1.0), (2, 300, 2, 1.0),
                                             (1, 640, 1, 8.0),   # peaked rows: the running maximum moves
                                             (5, 700, 8, 1.0),   # 120 two-tile units
                                             (3, 384, 4, 8.0),
                                             (8, 1000, 6, 1.0),  # 192 units: CTAs take two
                                             (16, 300, 12, 1.0),  # odd tile count: 384 units,
                                                                  # half without a second tile
                                             (4, 129, 3, 8.0),   # second tile of one row
                                             (6, 128, 2, 1.0)])  # one tile per sequence
def test_causal_attention(nseq, P, H_, q_std):
    Dh = 128
    d = H_ * Dh
    qkv_bits = synth.normal_bf16(531 + P, (nseq * P, 3 * d), 1.0)
    if q_std != 1.0:
        qkv_bits[:, :d] = synth.normal_bf16(532 + P, (nseq * P, d), q_std)
    out = torch.full((nseq * P, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    H.hydra_causal_attention(dev_bf16(qkv_bits), nseq, P, H_, Dh, out)
    x = f64(qkv_bits)
    got = host_f64(out)
    for s in range(nseq):
        blk = x[s * P:(s + 1) * P]
        q = blk[:, :d].reshape(P, H_, Dh)
        k = blk[:, d:2 * d].reshape(P, H_, Dh)
        v = blk[:, 2 * d:].reshape(P, H_, Dh)
        ref = O.causal_attention(q, k, v).reshape(P, d)
        assert_rel(got[s * P:(s + 1) * P], ref, TOL_LINEAR, f"attention seq {s}")


def test_causal_attention_strided_rows():
    """Row strides above 3d (qkv) and d (output): only the heads' columns of the output are
    written, each sequence's rows stay its own (the output is stored by sequence planes, so a
    partial last query tile writes nothing into the next sequence)."""
    nseq, P, H_, Dh = 3, 200, 2, 128
    d = H_ * Dh
    qkv_bits = synth.normal_bf16(537, (nseq * P, 3 * d + 64), 1.0)
    out = torch.full((nseq * P, d + 64), float("nan"), dtype=torch.bfloat16, device="cuda")
    H.hydra_causal_attention(dev_bf16(qkv_bits), nseq, P, H_, Dh, out)
    x = f64(qkv_bits)
    got = host_f64(out)
    assert np.isnan(got[:, d:]).all(), "columns past the heads were written"
    for s in range(nseq):
        blk = x[s * P:(s + 1) * P]
        q = blk[:, :d].reshape(P, H_, Dh)
        k = blk[:, d:2 * d].reshape(P, H_, Dh)
        v = blk[:, 2 * d:3 * d].reshape(P, H_, Dh)
        ref = O.causal_attention(q, k, v).reshape(P, d)
        assert_rel(got[s * P:(s + 1) * P, :d], ref, TOL_LINEAR, f"attention seq {s}")


def test_swiglu_residual_head_dot():
    R, F, d = 70, 520, 256
    gu = synth.normal_bf16(541, (R, 2 * F), 2.0)
    m = torch.empty(R, F, dtype=torch.bfloat16, device="cuda")
    H.hydra_swiglu(dev_bf16(gu), m)
    g = f64(gu)
    assert_rel(host_f64(m), O.round_bf16(O.swiglu(g[:, :F], g[:, F:])), TOL_LINEAR, "swiglu")

    h0 = synth.normal_f32(542, (R, d))
    y = synth.normal_bf16(543, (R, d))
    h = dev_f32(h0)
    H.hydra_residual_add(h, dev_bf16(y))
    assert_rel(host_f64(h), h0.astype(np.float64) + f64(y), 1e-6, "residual")

    x = synth.normal_bf16(544, (R, d))
    w = synth.normal_bf16(545, (d,), 0.02)
    out = torch.empty(R, device="cuda")
    H.hydra_head_dot(dev_bf16(x), dev_bf16(w), out)
    assert_rel(host_f64(out), f64(x) @ f64(w), 1e-5, "head dot")


# ------------------------------------------------------------------ the full pass


def make_model(cfg, seed, zero_B=False, lora_std=0.02, emb_std=1.0):
    nl, d, F, V, r = cfg["n_layers"], cfg["d_model"], cfg["ffn"], cfg["vocab"], cfg["lora_rank"]
    g = lambda i: synth.tensor_seed(seed, i)  # noqa: E731
    sep = {
        "wq": synth.normal_bf16(g(1), (nl, d, d), 0.02),
        "wk": synth.normal_bf16(g(2), (nl, d, d), 0.02),
        "wv": synth.normal_bf16(g(3), (nl, d, d), 0.02),
        "wo": synth.normal_bf16(g(4), (nl, d, d), 0.02),
        "wg": synth.normal_bf16(g(5), (nl, F, d), 0.02),
        "wu": synth.normal_bf16(g(6), (nl, F, d), 0.02),
        "wd": synth.normal_bf16(g(7), (nl, d, F), 0.02),
        "norm1": np.full((nl, d), ONE_BF16, dtype=np.uint16),
        "norm2": np.full((nl, d), ONE_BF16, dtype=np.uint16),
        "embed": synth.normal_bf16(g(8), (V, d), emb_std),
        "final_norm": np.full((d,), ONE_BF16, dtype=np.uint16),
        "lm_head": synth.normal_bf16(g(9), (V, d), 0.02),
        "w_rm": synth.normal_bf16(g(10), (d,), 0.02),
        "lora": {},
    }
    dims = {"wq": (d, d), "wv": (d, d), "wg": (F, d), "wu": (F, d), "wd": (d, F)}
    for i, (name, (n_out, n_in)) in enumerate(dims.items()):
        A = synth.normal_bf16(g(20 + i), (nl, r, n_in), lora_std)
        Bm = (np.zeros((nl, n_out, r), dtype=np.uint16) if zero_B
              else synth.normal_bf16(g(30 + i), (nl, n_out, r), lora_std))
        sep["lora"][name] = (A, Bm)
    w64 = {k: f64(v) for k, v in sep.items() if k != "lora"}
    w64["lora"] = {k: (f64(a), f64(b)) for k, (a, b) in sep["lora"].items()}
    return sep, w64


def oracle_cfg(cfg):
    return {"d": cfg["d_model"], "n_heads": cfg["n_heads"], "eps": cfg["rms_eps"],
            "lora_scale": cfg["lora_scale"], "rope_theta": cfg["rope_theta"],
            "n_layers": cfg["n_layers"]}


def run_pass(cfg, sep, ids, lengths):
    S = ids.shape[0]
    w = llama.to_device(llama.fuse_separate(sep), "cuda")
    ws = torch.empty(H.score_llama_workspace_size(cfg, S), dtype=torch.uint8, device="cuda")
    out = llama.alloc_outputs(S, cfg["response_len"], "cuda")
    H.hydra_score_llama(cfg, w, dev_i32(ids), None if lengths is None else dev_i32(lengths), ws, out)
    torch.cuda.synchronize()
    return {k: host_f64(v) for k, v in out.items()}


# Relative size of the fp32-accumulation difference that a kernel's stored values carry
# (measured: 0.23 % of the bf16 outputs of a K = 4096 tensor-core product differ by one ulp
# from the exactly rounded fp64 result, i.e. about 1e-5 relative before rounding).
DITHER_EPS = 1e-5


def chain_spread(w64, ids_s, P0, cfg, n):
    """How far two equally valid roundings of the bf16 chain drift apart: the oracle against
    itself with every stored value perturbed by DITHER_EPS relative before rounding."""
    kw = dict(seq_lengths=n, beta=cfg["beta"], gamma=cfg["gamma"], lam=cfg["lam"])
    O.set_storage_dither(DITHER_EPS, seed=17)
    try:
        alt = O.llama_score(w64, ids_s, P0, oracle_cfg(cfg), **kw)
    finally:
        O.set_storage_dither(0.0)
    return alt


def check_pass(cfg, got, w64, ids, lengths, derive_tol=False):
    """Compare a pass with the oracle. With derive_tol, each end-to-end tolerance is the
    larger of the stated one and 3x the chain's own spread under DITHER_EPS (a wide, deep
    bf16 chain amplifies one-ulp flips, so the stated per-kernel tolerances bound each
    kernel, not a composition of many)."""
    P0, L = cfg["prompt_len"], cfg["response_len"]
    g_, lam, beta = cfg["gamma"], cfg["lam"], cfg["beta"]
    S = ids.shape[0]
    e_r = e_v = 0.0
    for s in range(S):
        n = L if lengths is None else int(lengths[s])
        ref = O.llama_score(w64, ids[s], P0, oracle_cfg(cfg), seq_lengths=n, beta=beta,
                            gamma=g_, lam=lam)
        tol_lp, tol_lin = TOL_LOGP, TOL_LINEAR
        if derive_tol:
            alt = chain_spread(w64, ids[s], P0, cfg, n)
            spread_lp = max(max_abs_err(alt["logp_actor"], ref["logp_actor"]),
                            max_abs_err(alt["logp_ref"], ref["logp_ref"]))
            spread_lin = max(max_abs_err(alt["values"], ref["values"]),
                             abs(alt["score"] - ref["score"]))
            tol_lp = max(TOL_LOGP, 3 * spread_lp)
            tol_lin = max(TOL_LINEAR, 3 * spread_lin)
            mean_lp = lambda a, b: float(np.mean(np.abs(np.asarray(a)[:n] - np.asarray(b)[:n])))  # noqa: E731
            print(f"seq {s}: chain spread logp {spread_lp:.2e} (mean {mean_lp(alt['logp_actor'], ref['logp_actor']):.2e}), "
                  f"head {spread_lin:.2e} -> tolerances {tol_lp:.2e}, {tol_lin:.2e}; GPU mean logp "
                  f"error {mean_lp(got['logp_actor'][s], ref['logp_actor']):.2e}")
            print(f"seq {s}: GPU error logp actor {max_abs_err(got['logp_actor'][s], ref['logp_actor']):.2e}"
                  f", ref {max_abs_err(got['logp_ref'][s], ref['logp_ref']):.2e}, values "
                  f"{max_abs_err(got['values'][s], ref['values']):.2e}, score "
                  f"{abs(got['score'][s] - ref['score']):.2e} (stated logp tolerance {TOL_LOGP:.0e})")
        assert_abs(got["logp_actor"][s], ref["logp_actor"], tol_lp, f"logp_actor seq {s}")
        assert_abs(got["logp_ref"][s], ref["logp_ref"], tol_lp, f"logp_ref seq {s}")
        assert_rel(got["score"][s:s + 1], [ref["score"]], tol_lin, f"score seq {s}")
        assert_rel(got["values"][s], ref["values"], tol_lin, f"values seq {s}")
        # the KL part of the reward; the score enters at t = len - 1 on each side
        kl_got = got["reward"][s].copy()
        kl_ref = ref["reward"].copy()
        if n > 0:
            kl_got[n - 1] -= got["score"][s]
            kl_ref[n - 1] -= ref["score"]
        assert_abs(kl_got, kl_ref, tol_lp, f"KL reward seq {s}")
        e_r = max(e_r, max_abs_err(got["reward"][s], ref["reward"]))
        e_v = max(e_v, max_abs_err(got["values"][s], ref["values"]))
        # GAE on the GPU's own rewards and values: the scan's tolerance
        a1, r1 = O.gae(got["reward"][s:s + 1], got["values"][s:s + 1], [n], g_, lam)
        assert_rel(got["advantages"][s:s + 1], a1, TOL_GAE, f"advantages seq {s}")
        assert_rel(got["returns"][s:s + 1], r1, TOL_GAE, f"returns seq {s}")
        # end to end: reward and value errors pass through sum_k (gamma lambda)^k
        bound = (e_r + (1 + g_) * e_v) / (1 - g_ * lam) + TOL_GAE
        assert_abs(got["advantages"][s], ref["advantages"], bound, f"advantages e2e seq {s}")


SMALL = dict(n_layers=2, d_model=256, n_heads=2, head_dim=128, ffn=512, vocab=512,
             prompt_len=16, response_len=40, lora_rank=8, lora_scale=2.0, rms_eps=1e-6,
             rope_theta=10000.0, beta=0.1, gamma=1.0, lam=0.95)


def test_score_llama_small_ragged():
    cfg = dict(SMALL)
    sep, w64 = make_model(cfg, 61)
    S, P = 3, cfg["prompt_len"] + cfg["response_len"]
    ids = synth.randint(611, (S, P), 0, cfg["vocab"])
    lengths = np.array([40, 17, 1], dtype=np.int32)
    got = run_pass(cfg, sep, ids, lengths)
    check_pass(cfg, got, w64, ids, lengths)


def test_score_llama_several_key_blocks_rank16():
    cfg = dict(SMALL, n_layers=1, prompt_len=100, response_len=60, lora_rank=16, vocab=1024)
    sep, w64 = make_model(cfg, 62)
    ids = synth.randint(621, (2, 160), 0, cfg["vocab"])
    got = run_pass(cfg, sep, ids, None)
    check_pass(cfg, got, w64, ids, None)


@pytest.mark.parametrize("P0", [1, 2])
def test_score_llama_short_prompts_and_empty_response(P0):
    """Prompts of one token (the heads read every position: no compact last layer) and two
    tokens (the last layer drops one position per sequence), with an empty response among
    the sequences, against the oracle. Layer 0 forms its q/k/v products once for both streams
    in both cases."""
    cfg = dict(SMALL, prompt_len=P0)
    sep, w64 = make_model(cfg, 64 + P0)
    S, P = 3, cfg["prompt_len"] + cfg["response_len"]
    ids = synth.randint(641 + P0, (S, P), 0, cfg["vocab"])
    lengths = np.array([40, 0, 13], dtype=np.int32)
    got = run_pass(cfg, sep, ids, lengths)
    check_pass(cfg, got, w64, ids, lengths)
    assert got["score"][1] == 0.0 and not np.any(got["logp_actor"][1])


def test_score_llama_lora_off_streams_agree_bitwise():
    # §3 Dynamic LoRA: with every B = 0 the LoRA-on stream is the LoRA-off stream, so the
    # actor and reference log-probabilities agree exactly and the reward is the score alone
    cfg = dict(SMALL)
    sep, _ = make_model(cfg, 63, zero_B=True)
    S, P = 2, cfg["prompt_len"] + cfg["response_len"]
    ids = synth.randint(631, (S, P), 0, cfg["vocab"])
    lengths = np.array([40, 33], dtype=np.int32)
    got = run_pass(cfg, sep, ids, lengths)
    assert np.array_equal(got["logp_actor"], got["logp_ref"])
    expect = np.zeros_like(got["reward"])
    for s in range(S):
        expect[s, lengths[s] - 1] = got["score"][s]
    assert np.array_equal(got["reward"], expect)


def test_score_llama_full_width_one_layer():
    """Llama-7B widths (d 4096, 32 heads, FFN 11008, vocab 32000, LoRA r 16) at the
    benchmark's sequence shape (256 prompt + 512 response tokens), one decoder layer, one
    sequence, compared in full with the oracle."""
    cfg = dict(llama.LLAMA7B, n_layers=1)
    sep, w64 = make_model(cfg, 64)
    ids = synth.randint(641, (1, 768), 0, cfg["vocab"])
    lengths = np.array([512], dtype=np.int32)
    got = run_pass(cfg, sep, ids, lengths)
    check_pass(cfg, got, w64, ids, lengths, derive_tol=True)


def _dev_f64(t):
    """Exact fp64 values of a device bf16 tensor (bit copy to the host, widened by the oracle)."""
    return O.bf16_to_f64(t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16))


class _OracleLayers:
    """The oracle's per-layer weight arrays (exact fp64 values of the bf16 bits) taken from
    device weights in the fused layouts of hydra_score_llama, one decoder layer at a time: the
    first lookup of layer l splits and widens that layer and drops the one before it, since
    the fp64 copy of all 32 Llama-7B layers would need about 54 GB of host memory. Only tensors
    are sliced here; every value the oracle reads is a bf16 weight as the kernels see it."""

    def __init__(self, w, cfg):
        self.w, self.d, self.r = w, cfg["d_model"], cfg["lora_rank"]
        self.l, self.cache = None, None

    def layer(self, l):
        if self.l != l:
            self.cache = None
            W, d, r = self.w, self.d, self.r
            qkv = _dev_f64(W["w_qkv"][l])
            g_, u_ = llama.deinterleave_gate_up(_dev_f64(W["w_gu"][l]))
            a_qv, b_qkv = _dev_f64(W["a_qv"][l]), _dev_f64(W["b_qkv"][l])
            a_gu = _dev_f64(W["a_gu"][l])
            bg, bu = llama.deinterleave_gate_up(_dev_f64(W["b_gu"][l]))
            self.cache = {
                "wq": qkv[:d], "wk": qkv[d:2 * d], "wv": qkv[2 * d:], "wo": _dev_f64(W["w_o"][l]),
                "wg": g_, "wu": u_, "wd": _dev_f64(W["w_down"][l]),
                "norm1": _dev_f64(W["norm_attn"][l]), "norm2": _dev_f64(W["norm_ffn"][l]),
                ("A", "wq"): a_qv[:r], ("B", "wq"): b_qkv[:d, :r],
                ("A", "wv"): a_qv[r:], ("B", "wv"): b_qkv[2 * d:, r:],
                ("A", "wg"): a_gu[:r], ("B", "wg"): bg[:, :r],
                ("A", "wu"): a_gu[r:], ("B", "wu"): bu[:, r:],
                ("A", "wd"): _dev_f64(W["a_down"][l]), ("B", "wd"): _dev_f64(W["b_down"][l]),
            }
            self.l = l
        return self.cache


class _LayerItem:
    """weights[name][l] for the oracle, served by _OracleLayers."""

    def __init__(self, src, key):
        self.src, self.key = src, key

    def __getitem__(self, l):
        return self.src.layer(l)[self.key]


def oracle_view(w, cfg):
    src = _OracleLayers(w, cfg)
    v = {k: _LayerItem(src, k) for k in ("wq", "wk", "wv", "wo", "wg", "wu", "wd", "norm1", "norm2")}
    v["lora"] = {k: (_LayerItem(src, ("A", k)), _LayerItem(src, ("B", k)))
                 for k in ("wq", "wv", "wg", "wu", "wd")}
    for k in ("embed", "final_norm", "lm_head", "w_rm"):
        v[k] = _dev_f64(w[k])
    return v


def test_score_llama7b_32_layers_against_oracle():
    """The benchmark's model at its full depth: random-init Llama-7B (32 layers, d 4096, 32
    heads, FFN 11008, vocab 32000, LoRA r 16 on q/v/gate/up/down, s 2), drawn by the
    benchmark's generator and seed, on one sequence of 32 prompt + 64 response tokens,
    compared element by element with the oracle's 32-layer pass (scoring steps of Algorithm 1;
    §3 Dynamic LoRA; Appendix B's gamma and lambda). The log-probability tolerance is derived
    from the oracle's own spread under one-ulp storage dither at this depth, as in the
    one-layer full-width test; the stated per-kernel 5e-3 and the measured spread are printed
    beside the GPU error."""
    cfg = dict(llama.LLAMA7B, prompt_len=32, response_len=64)
    w = llama.random_device_weights(cfg, 4, "cuda")
    ids = synth.randint(4101, (1, 96), 0, cfg["vocab"])
    lengths = np.array([64], dtype=np.int32)
    ws = torch.empty(H.score_llama_workspace_size(cfg, 1), dtype=torch.uint8, device="cuda")
    out = llama.alloc_outputs(1, cfg["response_len"], "cuda")
    H.hydra_score_llama(cfg, w, dev_i32(ids), dev_i32(lengths), ws, out)
    torch.cuda.synchronize()
    got = {k: host_f64(v) for k, v in out.items()}
    check_pass(cfg, got, oracle_view(w, cfg), ids, lengths, derive_tol=True)
    del w, ws
    torch.cuda.empty_cache()


def test_score_llama7b_every_kernel_of_every_layer_against_oracle():
    """Every kernel of each of the 32 decoder layers of the benchmark's model at full width
    (Llama-7B shapes, LoRA r 16, the benchmark's generator and seed), on one sequence of 256
    prompt + 512 response tokens, against the oracle's step given the GPU's own input to that
    kernel, within the stated tolerance for linear outputs (2e-2 max(1, |ref|); the o and down
    projections are checked on what their epilogue added into the fp32 residual stream, the
    rotary outputs relative to the norm of each rotated pair, the SwiGLU output after the
    propagated one-ulp differences of its two unstored bf16 inputs). The
    layers run through the library's per-op entry points (the kernels
    and arguments hydra_score_llama launches, on every row of both streams), and the residual
    stream they leave equals, bit for bit, the one the full pass leaves in its workspace: after
    31 layers the whole stream (the workspace's first bytes; layer 0 there runs both streams
    from one accumulator), after layer 32 the rows the heads read (the pass runs its last
    layer's o projection and feed-forward block on those rows alone and keeps them where the
    q/k/v buffer was). So every kernel launch of the pass's decoder stack is checked at its own
    full size, without the drift that a chain of bf16 stages accumulates (steps of Algorithm
    1's scoring pass; §3 Dynamic LoRA: both streams). The pass's heads (final norm,
    log-probabilities of both streams, KL-penalised reward, score, values, GAE) are checked
    from the pass's own residual rows after layer 32 at their stated tolerances."""
    cfg = dict(llama.LLAMA7B)
    nl, d, F, r, nh = cfg["n_layers"], cfg["d_model"], cfg["ffn"], cfg["lora_rank"], cfg["n_heads"]
    P0, L = cfg["prompt_len"], cfg["response_len"]
    P, S = P0 + L, 1
    T = S * P
    s, eps, Dh = cfg["lora_scale"], cfg["rms_eps"], cfg["head_dim"]
    w = llama.random_device_weights(cfg, 4, "cuda")
    ids = torch.from_numpy(synth.randint(4201, (S, P), 0, cfg["vocab"])).cuda()
    bf = torch.bfloat16
    # the pass itself
    ws = torch.empty(H.score_llama_workspace_size(cfg, S), dtype=torch.uint8, device="cuda")
    out = llama.alloc_outputs(S, L, "cuda")
    H.hydra_score_llama(cfg, w, ids, None, ws, out)
    torch.cuda.synchronize()
    h_pass = ws[:2 * T * d * 4].view(torch.float32).view(2 * T, d).clone()
    # the last layer's residual rows: positions P0 - 1 .. P - 1 of each stream, kept in the
    # workspace after the residual stream h [2T, d] fp32 and the normed activations [2T, d] bf16
    up256 = lambda v: (v + 255) // 256 * 256  # noqa: E731
    Lc, off = L + 1, up256(2 * T * d * 4) + up256(2 * T * d * 2)
    hc_pass = ws[off:off + 2 * Lc * d * 4].view(torch.float32).view(2 * Lc, d).clone()
    # the same layers through the per-op entry points
    h = torch.empty(2 * T, d, device="cuda")
    H.hydra_embed(w["embed"], ids.view(-1), 2, h)
    table = torch.empty(P, Dh // 2, 2, device="cuda")
    H.hydra_rope_table(P, Dh, cfg["rope_theta"], table)
    a = torch.empty(2 * T, d, dtype=bf, device="cuda")
    qkv = torch.empty(2 * T, 3 * d, dtype=bf, device="cuda")
    attn = torch.empty(2 * T, d, dtype=bf, device="cuda")
    m = torch.empty(2 * T, F, dtype=bf, device="cuda")
    u2 = torch.empty(T, 2 * r, dtype=bf, device="cuda")
    u1 = torch.empty(T, r, dtype=bf, device="cuda")
    view = oracle_view(w, cfg)
    pos = np.arange(P)
    worst = {}

    def check(name, got, ref, scale=None, extra=None):
        # relative to max(1, |ref|), or to a given scale, after an allowed extra difference
        sc = np.maximum(1.0, np.abs(ref) if scale is None else scale)
        diff = np.abs(got - ref) if extra is None else np.maximum(np.abs(got - ref) - extra, 0.0)
        e = float(np.max(diff / sc))
        worst[name] = max(worst.get(name, 0.0), e)
        assert np.all(np.isfinite(got)), f"{name}, layer {l}: non-finite output"
        assert e <= TOL_LINEAR, f"{name}, layer {l}: max |err| / scale = {e:.3e} > {TOL_LINEAR:.0e}"

    def pair_norm(x):
        # rotary outputs: relative to the norm of each rotated pair (dims i, i + Dh/2 of a
        # head), which the rotation preserves; a one-ulp difference of the linear output
        # before the rotation is relative to that norm, not to the smaller rotated component
        y = x.reshape(T, nh, 2, Dh // 2)
        n = np.sqrt(y[:, :, 0] ** 2 + y[:, :, 1] ** 2)
        return np.concatenate([n, n], axis=-1).reshape(T, nh * Dh)

    for l in range(nl):
        if l == nl - 1:
            assert torch.equal(h, h_pass), "the per-op composition of 31 layers differs from the pass"
        lw = view["wq"][l]  # noqa: F841  (widens layer l's weights once)
        lo = view["lora"]
        h_in = host_f64(h)
        H.hydra_rmsnorm(h, w["norm_attn"][l], eps, a)
        H.hydra_lora_down(a[T:], w["a_qv"][l], s, u2)
        H.hydra_dual_linear_rope(a[:T], a[T:], w["w_qkv"][l], u2, w["b_qkv"][l], qkv[:T], qkv[T:],
                                 P, 2 * d, Dh, table)
        H.hydra_causal_attention(qkv, 2 * S, P, nh, Dh, attn)
        a1, g_u2, g_qkv, g_attn = host_f64(a), host_f64(u2), host_f64(qkv), host_f64(attn)
        H.hydra_dual_linear_ex(attn[:T], attn[T:], w["w_o"][l], None, None, h[:T], h[T:],
                               H.EPI_RESIDUAL)
        h_mid = host_f64(h)
        H.hydra_rmsnorm(h, w["norm_ffn"][l], eps, a)
        H.hydra_lora_down(a[T:], w["a_gu"][l], s, u2)
        H.hydra_dual_linear_ex(a[:T], a[T:], w["w_gu"][l], u2, w["b_gu"][l], m[:T], m[T:],
                               H.EPI_SWIGLU)
        H.hydra_lora_down(m[T:], w["a_down"][l], s, u1)
        H.hydra_dual_linear_ex(m[:T], m[T:], w["w_down"][l], u1, w["b_down"][l], h[:T], h[T:],
                               H.EPI_RESIDUAL)
        a2, g_ugu, g_m, g_ud, h_out = host_f64(a), host_f64(u2), host_f64(m), host_f64(u1), host_f64(h)

        # attention block, each kernel from its own GPU input
        check("rmsnorm (attention)", a1, O.round_bf16(O.rmsnorm(h_in, view["norm1"][l], eps)))
        A_q, A_v = lo["wq"][0][l], lo["wv"][0][l]
        check("lora_down q/v", g_u2, O.lora_down(a1[T:], np.concatenate([A_q, A_v]), s))
        q = O.dual_lora_linear(a1[:T], a1[T:], view["wq"][l], A_q, lo["wq"][1][l], s)
        k = O.dual_lora_linear(a1[:T], a1[T:], view["wk"][l], None, None, s)
        v = O.dual_lora_linear(a1[:T], a1[T:], view["wv"][l], A_v, lo["wv"][1][l], s)
        for i in range(2):
            rows = slice(i * T, (i + 1) * T)
            rq = O.round_bf16(O.rope(q[i].reshape(T, nh, Dh), pos, cfg["rope_theta"])).reshape(T, d)
            rk = O.round_bf16(O.rope(k[i].reshape(T, nh, Dh), pos, cfg["rope_theta"])).reshape(T, d)
            check("q/k/v linear + rotary, q", g_qkv[rows, :d], rq, pair_norm(rq))
            check("q/k/v linear + rotary, k", g_qkv[rows, d:2 * d], rk, pair_norm(rk))
            check("q/k/v linear, v", g_qkv[rows, 2 * d:], v[i])
            qq = g_qkv[rows, :d].reshape(T, nh, Dh)
            kk = g_qkv[rows, d:2 * d].reshape(T, nh, Dh)
            vv = g_qkv[rows, 2 * d:].reshape(T, nh, Dh)
            check("causal attention", g_attn[rows], O.round_bf16(O.causal_attention(qq, kk, vv)).reshape(T, d))
        o = O.dual_lora_linear(g_attn[:T], g_attn[T:], view["wo"][l], None, None, s)
        # the linear output (what the residual epilogue added), against the stated tolerance
        check("o linear (added into the residual stream)", h_mid - h_in, np.concatenate(o))
        # feed-forward block
        check("rmsnorm (feed-forward)", a2, O.round_bf16(O.rmsnorm(h_mid, view["norm2"][l], eps)))
        A_g, A_u = lo["wg"][0][l], lo["wu"][0][l]
        check("lora_down gate/up", g_ugu, O.lora_down(a2[T:], np.concatenate([A_g, A_u]), s))
        g_ = O.dual_lora_linear(a2[:T], a2[T:], view["wg"][l], A_g, lo["wg"][1][l], s)
        u_ = O.dual_lora_linear(a2[:T], a2[T:], view["wu"][l], A_u, lo["wu"][1][l], s)
        # the fused epilogue rounds gate and up to bf16 (as the oracle does) without storing
        # them: a one-ulp difference of either, which a different fp32 summation order may
        # give, reaches the SwiGLU output as |silu'(g) u| ulp(g) + |silu(g)| ulp(u)
        gg, uu = np.concatenate(g_), np.concatenate(u_)
        sig = 1.0 / (1.0 + np.exp(-gg))
        dsilu = sig * (1.0 + gg * (1.0 - sig))
        ulp = lambda x: np.exp2(np.floor(np.log2(np.maximum(np.abs(x), 1e-30))) - 7)  # noqa: E731
        check("gate/up linear + SwiGLU", g_m,
              np.concatenate([O.round_bf16(O.swiglu(g_[i], u_[i])) for i in range(2)]),
              extra=np.abs(dsilu * uu) * ulp(gg) + np.abs(gg * sig) * ulp(uu))
        check("lora_down down", g_ud, O.lora_down(g_m[T:], lo["wd"][0][l], s))
        dn = O.dual_lora_linear(g_m[:T], g_m[T:], view["wd"][l], lo["wd"][0][l], lo["wd"][1][l], s)
        check("down linear (added into the residual stream)", h_out - h_mid, np.concatenate(dn))
    h_rows = torch.cat([h[P0 - 1:P], h[T + P0 - 1:T + P]])
    assert torch.equal(h_rows, hc_pass), "the per-op composition's last layer differs from the pass"
    print("worst relative error per kernel over 32 layers (stated 2e-2): " +
          ", ".join(f"{k} {v:.1e}" for k, v in worst.items()))

    # the pass's heads from its own residual rows after layer 32 (llama_score's steps after
    # the decoder stack: final RMSNorm, LM head and log-softmax of both streams, KL-penalised
    # reward, score and values; GAE on the pass's own rewards and values), within the stated
    # tolerances: log-probabilities and the KL reward 5e-3, score and values 2e-2, GAE 1e-4
    hp = host_f64(hc_pass)  # row i of a stream: position P0 - 1 + i
    rows = np.arange(0, L)  # the hidden row that predicts each response token
    fin = [O.round_bf16(O.rmsnorm(hp[i * Lc:(i + 1) * Lc], view["final_norm"], eps)) for i in range(2)]
    resp = ids[0, P0:].cpu().numpy()
    lr, _ = O.log_softmax_gather(fin[0][rows] @ view["lm_head"].T, resp)
    la, _ = O.log_softmax_gather(fin[1][rows] @ view["lm_head"].T, resp)
    score = float(fin[0][Lc - 1] @ view["w_rm"])  # position P - 1, the last token
    values = fin[1][rows] @ view["w_rm"]
    reward = O.kl_penalised_reward(la[None], lr[None], [L], [score], cfg["beta"])[0]
    got = {k: v.cpu().double().numpy() for k, v in out.items()}
    heads = {
        "logp_actor": assert_abs(got["logp_actor"][0], la, TOL_LOGP, "logp_actor"),
        "logp_ref": assert_abs(got["logp_ref"][0], lr, TOL_LOGP, "logp_ref"),
        "reward": assert_abs(got["reward"][0], reward, TOL_LOGP, "KL-penalised reward"),
        "score": assert_rel(got["score"][:1], [score], TOL_LINEAR, "score"),
        "values": assert_rel(got["values"][0], values, TOL_LINEAR, "values"),
    }
    adv, ret = O.gae(got["reward"][:1], got["values"][:1], [L], cfg["gamma"], cfg["lam"])
    heads["advantages"] = assert_rel(got["advantages"][:1], adv, TOL_GAE, "advantages")
    heads["returns"] = assert_rel(got["returns"][:1], ret, TOL_GAE, "returns")
    print("heads from the pass's own residual stream: " +
          ", ".join(f"{k} {v:.1e}" for k, v in heads.items()))
    del w, ws
    torch.cuda.empty_cache()


# ------------------------------------------------------------------ full size, properties


@pytest.fixture(scope="module")
def llama7b():
    """The benchmark's model and batch: random-init Llama-7B (32 layers), 4 x (256 + 512)."""
    cfg = dict(llama.LLAMA7B)
    w = llama.random_device_weights(cfg, 4, "cuda")
    S, P = 4, cfg["prompt_len"] + cfg["response_len"]
    ids = torch.from_numpy(synth.randint(4001, (S, P), 0, cfg["vocab"])).cuda()
    ws = torch.empty(H.score_llama_workspace_size(cfg, S), dtype=torch.uint8, device="cuda")
    yield cfg, w, ids, ws
    del w, ws
    torch.cuda.empty_cache()


def _score(cfg, w, ids, lengths, ws):
    out = llama.alloc_outputs(ids.shape[0], cfg["response_len"], "cuda")
    H.hydra_score_llama(cfg, w, ids, lengths, ws, out)
    torch.cuda.synchronize()
    return {k: v.clone() for k, v in out.items()}


def test_llama7b_deterministic_batch_permutation_and_causal(llama7b):
    cfg, w, ids, ws = llama7b
    L = cfg["response_len"]
    lengths = torch.tensor([512, 300, 64, 1], dtype=torch.int32, device="cuda")
    a = _score(cfg, w, ids, lengths, ws)
    b = _score(cfg, w, ids, lengths, ws)
    for k in a:
        assert torch.equal(a[k], b[k]), f"{k} not deterministic"
    for k in ("logp_actor", "logp_ref", "reward", "values", "advantages"):
        assert torch.isfinite(a[k]).all()
    # sequences are independent: a permuted batch gives the permuted outputs, bit for bit
    perm = torch.tensor([2, 0, 3, 1], device="cuda")
    c = _score(cfg, w, ids[perm].contiguous(), lengths[perm].contiguous(), ws)
    for k in a:
        assert torch.equal(c[k], a[k][perm]), f"{k} changes with the batch order"
    # causal: changing sequence 0's last token moves nothing before it
    ids2 = ids.clone()
    ids2[0, -1] = (ids2[0, -1] + 1) % cfg["vocab"]
    d = _score(cfg, w, ids2, lengths, ws)
    for k in ("logp_actor", "logp_ref", "values"):
        assert torch.equal(d[k][0, :L - 1], a[k][0, :L - 1])
        assert torch.equal(d[k][1:], a[k][1:])
    assert not torch.equal(d["logp_actor"][0, L - 1], a["logp_actor"][0, L - 1])
    # GAE of the pass's own rewards and values (the scan's tolerance)
    rw, vv = host_f64(a["reward"]), host_f64(a["values"])
    adv, ret = O.gae(rw, vv, lengths.cpu().numpy(), cfg["gamma"], cfg["lam"])
    assert_rel(host_f64(a["advantages"]), adv, TOL_GAE, "advantages")
    assert_rel(host_f64(a["returns"]), ret, TOL_GAE, "returns")


def test_llama7b_lora_off_streams_agree_bitwise(llama7b):
    # §3 Dynamic LoRA at full size: zero every LoRA B and the two streams coincide
    cfg, w, ids, ws = llama7b
    wz = dict(w)
    for k in ("b_qkv", "b_gu", "b_down"):
        wz[k] = [torch.zeros_like(t) for t in w[k]]
    lengths = torch.tensor([512, 512, 200, 7], dtype=torch.int32, device="cuda")
    a = _score(cfg, wz, ids, lengths, ws)
    assert torch.equal(a["logp_actor"], a["logp_ref"])
    expect = torch.zeros_like(a["reward"])
    for s in range(4):
        expect[s, lengths[s] - 1] = a["score"][s]
    assert torch.equal(a["reward"], expect)


# ------------------------------------------------------------------ Hydra-PPO (three streams)


def _critic_set(cfg, seed):
    """A second LoRA set (the critic's): separate numpy bf16 bits and fp64 values."""
    sep2, w2 = make_model(cfg, seed)
    return sep2["lora"], w2["lora"]


def run_hydra_pass(cfg, sep, crit_sep, ids, lengths):
    S = ids.shape[0]
    w = llama.to_device(llama.fuse_separate(sep), "cuda")
    crit = llama.lora_to_device(llama.fuse_lora(crit_sep, cfg["d_model"], cfg["ffn"]), "cuda")
    ws = torch.empty(H.score_llama_hydra_workspace_size(cfg, S), dtype=torch.uint8, device="cuda")
    out = llama.alloc_outputs(S, cfg["response_len"], "cuda")
    H.hydra_score_llama_hydra(cfg, w, crit, dev_i32(ids),
                              None if lengths is None else dev_i32(lengths), ws, out)
    torch.cuda.synchronize()
    return {k: host_f64(v) for k, v in out.items()}


def test_score_llama_hydra_small_ragged():
    """Hydra-PPO's three-stream pass (critic LoRA set separate from the actor's) against the
    oracle's three-stream pass, sequence by sequence."""
    cfg = dict(SMALL)
    sep, w64 = make_model(cfg, 65)
    crit_sep, crit64 = _critic_set(cfg, 66)
    S, P = 3, cfg["prompt_len"] + cfg["response_len"]
    ids = synth.randint(651, (S, P), 0, cfg["vocab"])
    lengths = np.array([40, 23, 2], dtype=np.int32)
    got = run_hydra_pass(cfg, sep, crit_sep, ids, lengths)
    P0, L, g_, lam, beta = cfg["prompt_len"], cfg["response_len"], cfg["gamma"], cfg["lam"], cfg["beta"]
    for s in range(S):
        n = int(lengths[s])
        ref = O.llama_score_hydra(w64, crit64, ids[s], P0, oracle_cfg(cfg), seq_lengths=n,
                                  beta=beta, gamma=g_, lam=lam)
        assert_abs(got["logp_actor"][s], ref["logp_actor"], TOL_LOGP, f"logp_actor seq {s}")
        assert_abs(got["logp_ref"][s], ref["logp_ref"], TOL_LOGP, f"logp_ref seq {s}")
        assert_rel(got["score"][s:s + 1], [ref["score"]], TOL_LINEAR, f"score seq {s}")
        assert_rel(got["values"][s], ref["values"], TOL_LINEAR, f"values seq {s}")
        a1, r1 = O.gae(got["reward"][s:s + 1], got["values"][s:s + 1], [n], g_, lam)
        assert_rel(got["advantages"][s:s + 1], a1, TOL_GAE, f"advantages seq {s}")
    # the critic set moves the values: they differ from the J-Hydra pass's on-stream values
    jh = run_pass(cfg, sep, ids, lengths)
    assert np.array_equal(got["logp_actor"], jh["logp_actor"])
    assert np.array_equal(got["logp_ref"], jh["logp_ref"])
    assert np.max(np.abs(got["values"] - jh["values"])) > 1e-4


def test_score_llama_hydra_one_lora_set_is_j_hydra():
    """With the critic's LoRA set equal to the actor's, the three-stream pass returns the
    J-Hydra pass's outputs bit for bit."""
    cfg = dict(SMALL)
    sep, _ = make_model(cfg, 67)
    S, P = 2, cfg["prompt_len"] + cfg["response_len"]
    ids = synth.randint(671, (S, P), 0, cfg["vocab"])
    lengths = np.array([40, 31], dtype=np.int32)
    got = run_hydra_pass(cfg, sep, sep["lora"], ids, lengths)
    jh = run_pass(cfg, sep, ids, lengths)
    for k in got:
        assert np.array_equal(got[k], jh[k]), k
