"""Pins for the fp64 oracle: each oracle function is checked against something other than
itself -- hand-worked fixtures (tests/golden/), closed forms, invariants, brute force on
tiny inputs, or a library routine -- chosen so that a dropped term, a wrong sign, a wrong
index or a transposed operand fails at least one check."""
import json
import math
import os

import numpy as np
import pytest
import scipy.special

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


# ---------------------------------------------------------------- bf16 storage


def test_bf16_rounding_ties_to_even():
    one = 1.0
    ulp = 2.0 ** -7  # bf16 has 7 explicit mantissa bits
    assert O.round_bf16(np.array([one]))[0] == 1.0
    # exact half-ulp ties round to the even neighbour
    assert O.round_bf16(np.array([one + ulp / 2]))[0] == 1.0
    assert O.round_bf16(np.array([one + 3 * ulp / 2]))[0] == one + 2 * ulp
    # just above a tie rounds up
    assert O.round_bf16(np.array([one + ulp / 2 + 2.0 ** -20]))[0] == one + ulp
    assert O.f64_to_bf16_bits(np.array([1.0, -2.0]))[0] == 0x3F80
    assert O.f64_to_bf16_bits(np.array([1.0, -2.0]))[1] == 0xC000
    x = np.array([3.140625, -0.0078125, 65280.0])  # bf16-representable values
    assert np.array_equal(O.round_bf16(x), x)


# ---------------------------------------------------------------- a1/a2 LoRA linear


def test_lora_hand_example():
    g = _load("lora_dual_linear.json")
    x = np.array(g["x"], float)
    y_off, y_on = O.dual_lora_linear(x, x, np.array(g["W"], float), np.array(g["A"], float),
                                     np.array(g["B"], float), g["s"], out_bf16=False)
    assert np.array_equal(y_off, np.array(g["y_off"], float))
    assert np.array_equal(y_on, np.array(g["y_on"], float))


def _int_problem(rng, M, K, N, r):
    x = rng.integers(-3, 4, size=(M, K)).astype(float)
    W = rng.integers(-3, 4, size=(N, K)).astype(float)
    A = rng.integers(-2, 3, size=(r, K)).astype(float)
    B = rng.integers(-2, 3, size=(N, r)).astype(float)
    return x, W, A, B


def test_lora_brute_force_loops_nonsquare():
    # small integers: every product and sum is exact in fp64 and u is exact in bf16
    rng = np.random.default_rng(1)
    M, K, N, r, s = 5, 7, 3, 2, 2.0
    x, W, A, B = _int_problem(rng, M, K, N, r)
    x_off = x[::-1].copy()
    y_off, y_on = O.dual_lora_linear(x_off, x, W, A, B, s, out_bf16=False)
    for m in range(M):
        for n in range(N):
            acc_off = sum(x_off[m, k] * W[n, k] for k in range(K))
            acc = sum(x[m, k] * W[n, k] for k in range(K))
            for j in range(r):
                u = s * sum(x[m, k] * A[j, k] for k in range(K))
                acc += u * B[n, j]
            assert y_off[m, n] == acc_off
            assert y_on[m, n] == acc


def test_lora_equals_dense_merged_weight():
    # rank-r identity: x W^T + s (x A^T) B^T == x (W + s B A)^T
    rng = np.random.default_rng(2)
    x, W, A, B = _int_problem(rng, 6, 9, 4, 3)
    s = 0.5
    _, y_on = O.dual_lora_linear(x, x, W, A, B, s, out_bf16=False)
    dense = x @ (W + s * (B @ A)).T
    assert np.array_equal(y_on, dense)


def test_lora_off_switch_b_zero_and_s_zero():
    rng = np.random.default_rng(3)
    x = O.round_bf16(rng.standard_normal((8, 16)))
    W = O.round_bf16(0.02 * rng.standard_normal((12, 16)))
    A = O.round_bf16(0.02 * rng.standard_normal((4, 16)))
    B = np.zeros((12, 4))
    y_off, y_on = O.dual_lora_linear(x, x, W, A, B, 2.0)
    assert np.array_equal(y_off, y_on)
    B = O.round_bf16(0.02 * rng.standard_normal((12, 4)))
    y_off, y_on = O.dual_lora_linear(x, x, W, A, B, 0.0)
    assert np.array_equal(y_off, y_on)
    y_off2, y_on2 = O.dual_lora_linear(x, x, W, None, None, 2.0)
    assert np.array_equal(y_off2, y_on2) and np.array_equal(y_off2, y_off)


def test_lora_linear_in_s_and_bf16_output_rounding():
    rng = np.random.default_rng(4)
    x, W, A, B = _int_problem(rng, 4, 8, 5, 2)
    y1 = O.dual_lora_linear(x, x, W, A, B, 1.0, out_bf16=False)[1]
    y3 = O.dual_lora_linear(x, x, W, A, B, 3.0, out_bf16=False)[1]
    y0 = O.dual_lora_linear(x, x, W, A, B, 0.0, out_bf16=False)[1]
    assert np.array_equal(y3 - y0, 3.0 * (y1 - y0))
    xr = rng.standard_normal((4, 8))
    yb = O.dual_lora_linear(xr, xr, W, A, B, 1.0, out_bf16=True)[1]
    assert np.array_equal(O.round_bf16(yb), yb)


def test_lora_down_rounds_u_to_bf16():
    x = np.array([[1.0, 1.0]])
    A = np.array([[1.0, 2.0 ** -9]])  # s*(x A^T) = 1 + 2^-9: below half-ulp of bf16 at 1
    u = O.lora_down(x, A, 1.0)
    assert u[0, 0] == 1.0


# ---------------------------------------------------------------- a4 log-softmax + gather


def test_logsoftmax_hand_example():
    g = _load("logsoftmax_gather.json")
    base = np.log(np.array(g["z_is_log_of"], float))
    z = np.stack([base, base + g["shift_row1"]])
    logp, lse = O.log_softmax_gather(z, np.array(g["ids"]))
    np.testing.assert_allclose(logp, g["logp"], rtol=0, atol=1e-14)
    np.testing.assert_allclose(lse, g["lse"], rtol=0, atol=1e-14)


def test_logsoftmax_matches_scipy_and_invariants():
    rng = np.random.default_rng(5)
    T, V = 16, 257
    z = 3.0 * rng.standard_normal((T, V))
    ids = rng.integers(0, V, size=T)
    logp, lse = O.log_softmax_gather(z, ids)
    ref = scipy.special.log_softmax(z, axis=1)[np.arange(T), ids]
    np.testing.assert_allclose(logp, ref, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, scipy.special.logsumexp(z, axis=1), rtol=1e-14)
    # probabilities sum to one over the vocabulary
    np.testing.assert_allclose(np.exp(z - lse[:, None]).sum(1), 1.0, rtol=1e-12)
    # shift invariance per row
    c = rng.standard_normal(T)[:, None] * 50
    logp2, lse2 = O.log_softmax_gather(z + c, ids)
    np.testing.assert_allclose(logp2, logp, atol=1e-10)
    np.testing.assert_allclose(lse2, lse + c[:, 0], atol=1e-10)


def test_logsoftmax_special_cases():
    V = 1000
    z = np.full((2, V), 7.25)
    logp, _ = O.log_softmax_gather(z, np.array([0, V - 1]))
    np.testing.assert_allclose(logp, -math.log(V), atol=1e-13)
    logp1, lse1 = O.log_softmax_gather(np.array([[-3.5]]), np.array([0]))
    assert logp1[0] == 0.0 and lse1[0] == -3.5
    # brute force with exactly rounded sums on a tiny row
    row = np.array([0.3, -1.2, 2.5, 0.0])
    lse_bf = math.log(math.fsum(math.exp(v) for v in row))
    lp, ls = O.log_softmax_gather(row[None], np.array([1]))
    assert abs(ls[0] - lse_bf) < 1e-15 * 8 and abs(lp[0] - (row[1] - lse_bf)) < 1e-14


# ---------------------------------------------------------------- a5 KL-penalised reward


def test_kl_reward_hand_example():
    g = _load("kl_reward.json")
    r = O.kl_penalised_reward(np.array(g["logp_actor"]), np.array(g["logp_ref"]),
                              g["lengths"], g["score"], g["beta"])
    np.testing.assert_allclose(r, g["reward"], atol=1e-15)


def test_kl_reward_lora_off_gives_score_only_and_masking():
    rng = np.random.default_rng(6)
    S, L, V = 3, 5, 11
    z = rng.standard_normal((S * L, V))
    ids = rng.integers(0, V, size=S * L)
    lengths = np.array([5, 2, 0])
    score = np.array([1.5, -0.25, 9.0])
    out = O.token_logprobs_kl(z, z, ids, lengths, score, 0.1, S, L)
    expect = np.zeros((S, L))
    expect[0, 4] = 1.5
    expect[1, 1] = -0.25
    assert np.array_equal(out["reward"], expect)
    assert np.all(out["logp_actor"][1, 2:] == 0) and np.all(out["logp_ref"][2] == 0)
    # sign: actor more confident than reference at the sampled token -> negative penalty
    za = z.copy()
    za[np.arange(S * L), ids] += 2.0
    out2 = O.token_logprobs_kl(za, z, ids, lengths, None, 0.1, S, L)
    assert np.all(out2["reward"][0] < 0)


# ---------------------------------------------------------------- a7 GAE


def test_gae_hand_examples():
    g = _load("gae.json")
    for c in g["cases"]:
        adv, ret = O.gae(np.array(c["rewards"]), np.array(c["values"]), c["lengths"],
                         c["gamma"], c["lam"])
        np.testing.assert_allclose(adv, c["advantages"], atol=1e-15)
        np.testing.assert_allclose(ret, c["returns"], atol=1e-15)


def _gae_problem(seed, S=4, L=37):
    rng = np.random.default_rng(seed)
    r = rng.standard_normal((S, L))
    v = rng.standard_normal((S, L))
    lengths = np.array([L, L // 2, 1, 0])[:S]
    return r, v, lengths


def test_gae_gamma_lambda_one_is_return_minus_value():
    r, v, lengths = _gae_problem(7)
    adv, ret = O.gae(r, v, lengths, 1.0, 1.0)
    for s, n in enumerate(lengths):
        for t in range(n):
            assert abs(adv[s, t] - (math.fsum(r[s, t:n]) - v[s, t])) < 1e-12
        assert np.all(adv[s, n:] == 0) and np.all(ret[s, n:] == 0)


def test_gae_lambda_zero_is_td_residual_and_returns():
    r, v, lengths = _gae_problem(8)
    gamma = 0.9
    adv, ret = O.gae(r, v, lengths, gamma, 0.0)
    for s, n in enumerate(lengths):
        for t in range(n):
            vn = v[s, t + 1] if t + 1 < n else 0.0
            assert abs(adv[s, t] - (r[s, t] + gamma * vn - v[s, t])) < 1e-14
    np.testing.assert_allclose(ret, np.where(adv != 0, adv + v, 0.0), atol=1e-14)


def test_gae_direct_sum_definition():
    # A_t = sum_l (gamma lambda)^l delta_{t+l} (GAE as an exponentially weighted sum)
    r, v, lengths = _gae_problem(9)
    gamma, lam = 0.97, 0.95
    adv, ret = O.gae(r, v, lengths, gamma, lam)
    for s, n in enumerate(lengths):
        delta = [r[s, t] + gamma * (v[s, t + 1] if t + 1 < n else 0.0) - v[s, t] for t in range(n)]
        for t in range(n):
            ref = math.fsum(((gamma * lam) ** l) * delta[t + l] for l in range(n - t))
            assert abs(adv[s, t] - ref) < 1e-12
            assert abs(ret[s, t] - (ref + v[s, t])) < 1e-12


def test_gae_geometric_closed_form():
    L, lam, c = 50, 0.95, 0.7
    r = np.full((1, L), c)
    adv, _ = O.gae(r, np.zeros((1, L)), [L], 1.0, lam)
    for t in range(L):
        n = L - t
        assert abs(adv[0, t] - c * (1 - lam ** n) / (1 - lam)) < 1e-12


# ---------------------------------------------------------------- a8 Llama pieces


def test_rmsnorm_definition():
    h = np.array([[3.0, 4.0], [0.0, 2.0]])
    out = O.rmsnorm(h, np.array([1.0, 2.0]), 0.0)
    np.testing.assert_allclose(out[0], [3 / math.sqrt(12.5), 8 / math.sqrt(12.5)], rtol=1e-15)
    np.testing.assert_allclose(out[1], [0.0, 4 / math.sqrt(2.0)], rtol=1e-15)
    out_eps = O.rmsnorm(np.zeros((1, 4)), np.ones(4), 1e-6)
    assert np.all(out_eps == 0)


def test_rope_against_rotation_matrices():
    rng = np.random.default_rng(10)
    T, H, D, theta = 5, 2, 8, 10000.0
    x = rng.standard_normal((T, H, D))
    pos = np.array([0, 1, 2, 7, 100])
    y = O.rope(x, pos, theta)
    half = D // 2
    for t in range(T):
        for h in range(H):
            for i in range(half):
                ang = pos[t] * theta ** (-2.0 * i / D)
                R = np.array([[math.cos(ang), -math.sin(ang)], [math.sin(ang), math.cos(ang)]])
                ref = R @ np.array([x[t, h, i], x[t, h, i + half]])
                assert abs(y[t, h, i] - ref[0]) < 1e-12 and abs(y[t, h, i + half] - ref[1]) < 1e-12
    np.testing.assert_allclose(y[0], x[0], atol=0)  # position 0 is the identity
    # relative-position property: <rope(q, m), rope(k, n)> depends on m - n only
    q = rng.standard_normal((1, 1, D))
    k = rng.standard_normal((1, 1, D))
    d1 = np.sum(O.rope(q, [9], theta) * O.rope(k, [4], theta))
    d2 = np.sum(O.rope(q, [25], theta) * O.rope(k, [20], theta))
    assert abs(d1 - d2) < 1e-12


def test_causal_attention_brute_force_and_causality():
    rng = np.random.default_rng(11)
    T, H, D = 6, 2, 4
    q, k, v = (rng.standard_normal((T, H, D)) for _ in range(3))
    out = O.causal_attention(q, k, v)
    for h in range(H):
        for i in range(T):
            sc = [sum(q[i, h, d] * k[j, h, d] for d in range(D)) / math.sqrt(D) for j in range(i + 1)]
            mx = max(sc)
            w = [math.exp(s_ - mx) for s_ in sc]
            tot = math.fsum(w)
            ref = [math.fsum(w[j] * v[j, h, d] for j in range(i + 1)) / tot for d in range(D)]
            np.testing.assert_allclose(out[i, h], ref, atol=1e-12)
    np.testing.assert_allclose(out[0], v[0], atol=1e-15)  # first query sees only itself
    k2, v2 = k.copy(), v.copy()
    k2[4:] += 10.0
    v2[4:] -= 3.0
    out2 = O.causal_attention(q, k2, v2)
    np.testing.assert_allclose(out2[:4], out[:4], atol=0)


def test_swiglu_against_scipy():
    rng = np.random.default_rng(12)
    g, u = rng.standard_normal(50) * 4, rng.standard_normal(50)
    np.testing.assert_allclose(O.swiglu(g, u), g * scipy.special.expit(g) * u, rtol=1e-13)
    assert O.swiglu(np.array([0.0]), np.array([5.0]))[0] == 0.0


# ---------------------------------------------------------------- composition invariants


def tiny_llama(seed=13, n_layers=2, d=32, H=4, F=48, V=64, r=4, zero_B=False):
    rng = np.random.default_rng(seed)
    bf = lambda *shape, std=0.02: O.round_bf16(std * rng.standard_normal(shape))  # noqa: E731
    w = {
        "embed": bf(V, d, std=1.0),
        "wq": bf(n_layers, d, d), "wk": bf(n_layers, d, d), "wv": bf(n_layers, d, d),
        "wo": bf(n_layers, d, d), "wg": bf(n_layers, F, d), "wu": bf(n_layers, F, d),
        "wd": bf(n_layers, d, F),
        "norm1": np.ones((n_layers, d)), "norm2": np.ones((n_layers, d)),
        "final_norm": np.ones(d), "lm_head": bf(V, d, std=0.2), "w_rm": bf(d, std=0.2),
        "lora": {},
    }
    dims = {"wq": (d, d), "wv": (d, d), "wg": (F, d), "wu": (F, d), "wd": (d, F)}
    for name, (n_out, n_in) in dims.items():
        A = bf(n_layers, r, n_in, std=0.2)
        B = np.zeros((n_layers, n_out, r)) if zero_B else bf(n_layers, n_out, r, std=0.2)
        w["lora"][name] = (A, B)
    cfg = {"d": d, "n_heads": H, "eps": 1e-6, "lora_scale": 2.0, "rope_theta": 10000.0,
           "n_layers": n_layers}
    return w, cfg


def test_llama_score_lora_off_invariants():
    w, cfg = tiny_llama(zero_B=True)
    rng = np.random.default_rng(14)
    ids = rng.integers(0, 64, size=12)
    out = O.llama_score(w, ids, 4, cfg)
    assert np.array_equal(out["h_off"], out["h_on"])
    assert np.array_equal(out["logp_actor"], out["logp_ref"])
    expect_r = np.zeros(8)
    expect_r[-1] = out["score"]
    assert np.array_equal(out["reward"], expect_r)
    adv, ret = O.gae(out["reward"][None], out["values"][None], [8], 1.0, 0.95)
    np.testing.assert_allclose(out["advantages"], adv[0], atol=0)


def test_llama_score_causal_and_lora_changes_actor_only():
    w, cfg = tiny_llama()
    rng = np.random.default_rng(15)
    ids = rng.integers(0, 64, size=12)
    out = O.llama_score(w, ids, 4, cfg)
    ids2 = ids.copy()
    ids2[-1] = (ids2[-1] + 1) % 64
    out2 = O.llama_score(w, ids2, 4, cfg)
    # hidden states before the last position do not see the changed last token
    np.testing.assert_allclose(out2["h_off"][:-1], out["h_off"][:-1], atol=0)
    np.testing.assert_allclose(out2["h_on"][:-1], out["h_on"][:-1], atol=0)
    w0, _ = tiny_llama(zero_B=True)
    ref0 = O.llama_score(w0, ids, 4, cfg)
    # turning LoRA on changes the actor stream but never the reference stream
    np.testing.assert_allclose(out["logp_ref"], ref0["logp_ref"], atol=0)
    assert np.max(np.abs(out["logp_actor"] - ref0["logp_actor"])) > 1e-6


@pytest.mark.parametrize("n", [8, 5, 0])
def test_llama_score_heads_read_only_the_last_prompt_position_on(monkeypatch, n):
    """The heads (log-probabilities of both streams, values, reward score) read the final
    hidden states only at positions P - 1 .. T - 1 of the sequence: the rows that predict the
    response tokens and the last token's row (Alg. 1 scoring steps). Overwriting every other
    row changes no output. The GPU pass relies on this reading when it runs its last layer's
    o projection and feed-forward block on those rows alone."""
    w, cfg = tiny_llama()
    rng = np.random.default_rng(16)
    ids = rng.integers(0, 64, size=12)
    P = 4
    ref = O.llama_score(w, ids, P, cfg, seq_lengths=n)
    real = O.llama_final_hidden

    def scrambled(weights, ids_, cfg_, n_layers=None):
        f_off, f_on = real(weights, ids_, cfg_, n_layers)
        junk = np.random.default_rng(17).standard_normal((P - 1, f_off.shape[1]))
        f_off, f_on = f_off.copy(), f_on.copy()
        f_off[:P - 1] = junk
        f_on[:P - 1] = -junk
        return f_off, f_on

    monkeypatch.setattr(O.hydra_oracle, "llama_final_hidden", scrambled)
    out = O.llama_score(w, ids, P, cfg, seq_lengths=n)
    for k in ("logp_actor", "logp_ref", "reward", "values", "advantages", "returns"):
        assert np.array_equal(out[k], ref[k]), k
    assert out["score"] == ref["score"]
    assert not np.array_equal(out["h_off"], ref["h_off"])


def test_storage_dither_is_off_by_default_and_bounded():
    x = np.array([1.0, 1.0 + 2 ** -9 + 2 ** -20, 3.0, -0.3])
    base = O.round_bf16(x)
    O.set_storage_dither(1e-5, seed=1)
    try:
        d = O.round_bf16(x)
        # a dither far below half an ulp moves a value only when it sits next to a tie
        assert np.array_equal(d[[0, 2]], base[[0, 2]])
        assert np.all(np.abs(d - base) <= 2 ** -7 * np.abs(base))
    finally:
        O.set_storage_dither(0.0)
    assert np.array_equal(O.round_bf16(x), base)


def test_hydra_ppo_one_lora_set_is_j_hydra():
    """Hydra-PPO with the critic's LoRA set equal to the actor's is J-Hydra-PPO (§3: J-Hydra
    uses one LoRA set for actor and critic): every output equals llama_score's exactly."""
    w, cfg = tiny_llama()
    ids = np.random.default_rng(16).integers(0, 64, size=12)
    j = O.llama_score(w, ids, 4, cfg, seq_lengths=6)
    h = O.llama_score_hydra(w, w["lora"], ids, 4, cfg, seq_lengths=6)
    for k in ("logp_actor", "logp_ref", "reward", "values", "advantages", "returns"):
        assert np.array_equal(h[k], j[k]), k
    assert h["score"] == j["score"]
    assert np.array_equal(h["h_crit"], j["h_on"]) and np.array_equal(h["h_act"], j["h_on"])


def test_hydra_ppo_critic_stream_is_separate():
    """The critic's LoRA set moves only the values: with its B = 0 the critic stream is the
    LoRA-off stream (values = w_rm . h_off rows); a different critic set leaves the actor and
    reference log-probabilities, the score and the reward unchanged."""
    w, cfg = tiny_llama()
    w0, _ = tiny_llama(zero_B=True)
    ids = np.random.default_rng(17).integers(0, 64, size=12)
    off_crit = O.llama_score_hydra(w, w0["lora"], ids, 4, cfg)
    assert np.array_equal(off_crit["h_crit"], off_crit["h_off"])
    rows = np.arange(3, 11)
    assert np.array_equal(off_crit["values"], off_crit["h_off"][rows] @ w["w_rm"])
    other, _ = tiny_llama(seed=99)
    alt = O.llama_score_hydra(w, other["lora"], ids, 4, cfg)
    for k in ("logp_actor", "logp_ref", "reward"):
        assert np.array_equal(alt[k], off_crit[k]), k
    assert alt["score"] == off_crit["score"]
    assert np.max(np.abs(alt["values"] - off_crit["values"])) > 1e-6


# ------------------------------------------------------------------ PPO update-side losses


def test_ppo_loss_hand_example():
    # eps = 0.2; ratios 0.5, 1.0, 1.5 (logp_new - logp_old = log r), advantages +1, -2, +1
    lo = np.zeros((1, 3))
    ln = np.log(np.array([[0.5, 1.0, 1.5]]))
    A = np.array([[1.0, -2.0, 1.0]])
    R = np.array([[1.0, 2.0, 3.0]])
    V = np.array([[1.5, 2.0, 1.0]])
    out = O.ppo_loss(ln, lo, A, R, V, [3], clip_eps=0.2)
    # s = min(0.5, 0.8) = 0.5; min(-2, -2) = -2; min(1.5, 1.2) = 1.2
    assert abs(out["loss_clip"] - (-(0.5 - 2.0 + 1.2) / 3)) < 1e-15
    assert abs(out["loss_value"] - (0.25 + 0.0 + 4.0) / 3) < 1e-15
    assert out["clip_frac"] == 2 / 3
    np.testing.assert_allclose(out["grad_logp"], [[-0.5 / 3, 2.0 / 3, 0.0]], atol=1e-15)
    np.testing.assert_allclose(out["grad_values"], [[1.0 / 3, 0.0, -4.0 / 3]], atol=1e-15)


def _ppo_problem(seed, S=3, L=11):
    rng = np.random.default_rng(seed)
    lo = rng.normal(-2.0, 0.5, (S, L))
    ln = lo + rng.normal(0.0, 0.3, (S, L))
    A = rng.normal(0.0, 1.5, (S, L))
    R = rng.normal(0.0, 1.0, (S, L))
    V = rng.normal(0.0, 1.0, (S, L))
    lengths = np.array([L, 5, 0][:S])
    return ln, lo, A, R, V, lengths


@pytest.mark.parametrize("whiten", [False, True])
def test_ppo_loss_gradients_match_finite_differences(whiten):
    ln, lo, A, R, V, lengths = _ppo_problem(21)
    out = O.ppo_loss(ln, lo, A, R, V, lengths, whiten=whiten)
    h = 1e-6
    for s, t in [(0, 0), (0, 7), (1, 3), (1, 6), (2, 1)]:
        lp, lm = ln.copy(), ln.copy()
        lp[s, t] += h
        lm[s, t] -= h
        fd = (O.ppo_loss(lp, lo, A, R, V, lengths, whiten=whiten)["loss_clip"] -
              O.ppo_loss(lm, lo, A, R, V, lengths, whiten=whiten)["loss_clip"]) / (2 * h)
        assert abs(fd - out["grad_logp"][s, t]) < 1e-7, (s, t)
        vp, vm = V.copy(), V.copy()
        vp[s, t] += h
        vm[s, t] -= h
        fd = (O.ppo_loss(ln, lo, A, R, vp, lengths)["loss_value"] -
              O.ppo_loss(ln, lo, A, R, vm, lengths)["loss_value"]) / (2 * h)
        assert abs(fd - out["grad_values"][s, t]) < 1e-7, (s, t)


def test_ppo_loss_special_cases():
    ln, lo, A, R, V, lengths = _ppo_problem(22)
    valid = np.arange(11)[None, :] < lengths[:, None]
    # policy unchanged: ratio 1, L^CLIP is the mean advantage, nothing clipped, KL 0
    same = O.ppo_loss(lo, lo, A, R, V, lengths)
    assert abs(same["loss_clip"] + A[valid].mean()) < 1e-12
    assert same["clip_frac"] == 0.0 and same["approx_kl"] == 0.0
    # whitened advantages have mean 0 and variance 1 over the valid tokens
    w = O.ppo_loss(lo, lo, A, R, V, lengths, whiten=True)
    assert abs(w["loss_clip"]) < 1e-12
    assert abs(w["adv_mean"] - A[valid].mean()) < 1e-12 and abs(w["adv_std"] - A[valid].std()) < 1e-12
    # a huge ratio with positive advantage is clipped: no gradient
    big = lo.copy()
    big[0, 0] += 5.0
    g = O.ppo_loss(big, lo, np.abs(A), R, V, lengths)
    assert g["grad_logp"][0, 0] == 0.0
    # no valid tokens
    z = O.ppo_loss(ln, lo, A, R, V, [0, 0, 0])
    assert z["loss_clip"] == 0.0 and not z["grad_logp"].any()


def test_ppo_loss_shards_with_merged_moments_add_up():
    # a batch split into two shards, each normalised by the whole batch's moments: the
    # shards' losses add up to the whole batch's and their gradients are the whole's rows
    ln, lo, A, R, V, lengths = _ppo_problem(23, S=3, L=11)
    for whiten in (False, True):
        full = O.ppo_loss(ln, lo, A, R, V, lengths, whiten=whiten)
        valid = np.arange(11)[None, :] < lengths[:, None]
        mom = (valid.sum(), A[valid].mean(), ((A[valid] - A[valid].mean()) ** 2).sum())
        p0 = O.ppo_loss(ln[:1], lo[:1], A[:1], R[:1], V[:1], lengths[:1], whiten=whiten, moments=mom)
        p1 = O.ppo_loss(ln[1:], lo[1:], A[1:], R[1:], V[1:], lengths[1:], whiten=whiten, moments=mom)
        for k in ("loss_clip", "loss_value", "clip_frac", "approx_kl"):
            assert abs(p0[k] + p1[k] - full[k]) < 1e-12, k
        np.testing.assert_allclose(np.vstack([p0["grad_logp"], p1["grad_logp"]]), full["grad_logp"],
                                   atol=1e-15)


# ------------------------------------------------------------------ generation


def test_gumbel_argmax_draws_follow_softmax():
    """The Gumbel-max trick: argmax(z + g), g standard Gumbel, is a draw from softmax(z).
    200k draws with numpy's own Gumbel noise: every empirical frequency within 5 sigma."""
    z = np.array([1.5, -0.5, 0.0, 2.2, -3.0])
    p = scipy.special.softmax(z)
    rng = np.random.default_rng(5)
    N = 200_000
    g = -np.log(-np.log(rng.random((N, z.size))))
    counts = np.bincount(np.argmax(z + g, axis=1), minlength=z.size)
    draws = np.array([O.gumbel_argmax(z, g[i]) for i in range(2000)])
    assert np.array_equal(draws, np.argmax(z + g[:2000], axis=1))
    sigma = np.sqrt(N * p * (1 - p))
    assert np.all(np.abs(counts - N * p) < 5 * sigma), (counts, N * p)
    assert O.gumbel_argmax(z) == 3
    assert O.gumbel_argmax(np.array([1.0, 3.0, 3.0])) == 1  # ties: lowest index


@pytest.mark.parametrize("noise", [False, True])
def test_generate_is_the_scoring_pass_on_its_own_sequence(noise):
    """Each step's distribution is that of the last position of a full causal pass: the
    recorded log-probs, values and score equal llama_score's on the finished sequence, and
    every token is the argmax of that position's actor logits plus the step's noise."""
    w, cfg = tiny_llama(seed=21)
    rng = np.random.default_rng(22)
    prompt = rng.integers(0, 64, size=5)
    n = 7
    g = -np.log(-np.log(rng.random((n, 64)))) if noise else None
    gen = O.llama_generate(w, prompt, n, cfg, gumbel=g)
    seq = np.concatenate([prompt, gen["tokens"]])
    ref = O.llama_score(w, seq, 5, cfg)
    for k in ("logp_actor", "logp_ref", "values"):
        np.testing.assert_allclose(gen[k], ref[k], rtol=0, atol=1e-12)
    assert abs(gen["score"] - ref["score"]) < 1e-12
    z_on = ref["h_on"][4:4 + n] @ w["lm_head"].T
    expect = np.argmax(z_on + (0.0 if g is None else g), axis=1)
    assert np.array_equal(gen["tokens"], expect)
    # log-probabilities are normalised distributions' entries
    assert np.all(gen["logp_actor"] <= 0) and np.all(gen["logp_ref"] <= 0)


def test_generate_lora_off_streams_agree():
    w, cfg = tiny_llama(seed=23, zero_B=True)
    prompt = np.random.default_rng(24).integers(0, 64, size=3)
    gen = O.llama_generate(w, prompt, 4, cfg)
    np.testing.assert_array_equal(gen["logp_actor"], gen["logp_ref"])


def _torch_final_hidden(w, ids, cfg):
    """The decoder stack written with PyTorch library operations in fp64: F.linear,
    F.rms_norm, the causal F.scaled_dot_product_attention, F.silu, and the rotary
    embedding as a complex rotation of the pairs (i, i + D/2). LoRA on wq/wv/wg/wu/wd of the
    LoRA-on stream only."""
    import torch
    import torch.nn.functional as F
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.float64))  # noqa: E731
    d, H, eps, s = cfg["d"], cfg["n_heads"], cfg["eps"], cfg["lora_scale"]
    Dh, T = d // H, len(ids)
    inv = cfg["rope_theta"] ** (-torch.arange(Dh // 2, dtype=torch.float64) * 2.0 / Dh)
    ang = torch.arange(T, dtype=torch.float64)[:, None] * inv[None, :]
    rot = torch.polar(torch.ones_like(ang), ang)[:, None, :]  # [T, 1, Dh/2]

    def rope(x):
        z = torch.complex(x[..., :Dh // 2], x[..., Dh // 2:]) * rot
        return torch.cat([z.real, z.imag], dim=-1)

    def lin(x, name, l, on):
        y = F.linear(x, t(w[name][l]))
        if on and name in w["lora"]:
            A, B = w["lora"][name]
            y = y + s * F.linear(F.linear(x, t(A[l])), t(B[l]))
        return y

    outs = []
    for on in (False, True):
        h = t(w["embed"])[torch.as_tensor(np.asarray(ids))]
        for l in range(cfg["n_layers"]):
            a = F.rms_norm(h, (d,), weight=t(w["norm1"][l]), eps=eps)
            q = rope(lin(a, "wq", l, on).view(T, H, Dh)).transpose(0, 1)
            k = rope(lin(a, "wk", l, on).view(T, H, Dh)).transpose(0, 1)
            v = lin(a, "wv", l, on).view(T, H, Dh).transpose(0, 1)
            att = F.scaled_dot_product_attention(q, k, v, is_causal=True).transpose(0, 1).reshape(T, d)
            h = h + lin(att, "wo", l, on)
            a = F.rms_norm(h, (d,), weight=t(w["norm2"][l]), eps=eps)
            h = h + lin(F.silu(lin(a, "wg", l, on)) * lin(a, "wu", l, on), "wd", l, on)
        outs.append(F.rms_norm(h, (d,), weight=t(w["final_norm"]), eps=eps).numpy())
    return outs


def test_llama_composition_matches_a_library_forward(monkeypatch):
    """The whole decoder stack (embedding, RMSNorm, rotary q/k, causal attention, residuals,
    SwiGLU, LoRA on the on stream, final norm) against the same architecture built from
    PyTorch's library operations. The bf16 storage rounding is switched off in the oracle
    for this comparison, so both sides are exact fp64 compositions."""
    pytest.importorskip("torch")
    w, cfg = tiny_llama(seed=31, n_layers=3, d=32, H=4, F=48, V=64, r=4)
    rng = np.random.default_rng(32)
    w["norm1"] = 0.5 + rng.random(w["norm1"].shape)
    w["norm2"] = 0.5 + rng.random(w["norm2"].shape)
    w["final_norm"] = 0.5 + rng.random(w["final_norm"].shape)
    ids = rng.integers(0, 64, size=13)
    ref_off, ref_on = _torch_final_hidden(w, ids, cfg)
    monkeypatch.setattr(O.hydra_oracle, "round_bf16", lambda x: np.asarray(x, dtype=np.float64))
    f_off, f_on = O.llama_final_hidden(w, ids, cfg)
    np.testing.assert_allclose(f_off, ref_off, rtol=1e-9, atol=1e-10)
    np.testing.assert_allclose(f_on, ref_on, rtol=1e-9, atol=1e-10)
    assert not np.allclose(f_off, f_on)  # the LoRA term reaches the on stream


def test_hydra_three_stream_composition_matches_a_library_forward(monkeypatch):
    """The three-stream stack of the Hydra-PPO oracle (LoRA off, the actor's set, the critic's
    set) against the library forward of each stream, bf16 storage rounding switched off."""
    pytest.importorskip("torch")
    w, cfg = tiny_llama(seed=41, n_layers=2, d=32, H=4, F=48, V=64, r=4)
    wc, _ = tiny_llama(seed=42, n_layers=2, d=32, H=4, F=48, V=64, r=4)
    rng = np.random.default_rng(43)
    w["norm1"] = 0.5 + rng.random(w["norm1"].shape)
    w["norm2"] = 0.5 + rng.random(w["norm2"].shape)
    w["final_norm"] = 0.5 + rng.random(w["final_norm"].shape)
    ids = rng.integers(0, 64, size=11)
    ref_off, ref_act = _torch_final_hidden(w, ids, cfg)
    _, ref_crit = _torch_final_hidden(dict(w, lora=wc["lora"]), ids, cfg)
    monkeypatch.setattr(O.hydra_oracle, "round_bf16", lambda x: np.asarray(x, dtype=np.float64))
    out = O.llama_score_hydra(w, wc["lora"], ids, 4, cfg)
    np.testing.assert_allclose(out["h_off"], ref_off, rtol=1e-9, atol=1e-10)
    np.testing.assert_allclose(out["h_act"], ref_act, rtol=1e-9, atol=1e-10)
    np.testing.assert_allclose(out["h_crit"], ref_crit, rtol=1e-9, atol=1e-10)
