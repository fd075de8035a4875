"""fp64 CPU oracle for the Hydra-PPO experience-scoring path (arXiv 2309.00754).

TEST INFRASTRUCTURE, NOT PRODUCT CODE. Only the test-suite, the package's smoke check
and the benchmark's CPU-baseline leg may import this module. The CUDA library never
calls it, and it shares no code with the CUDA library: no kernels, helpers, tables or
constants. Inputs arrive as plain numpy arrays (bf16 tensors as uint16 bit patterns).

Everything is computed in float64 from the exact input values. Where the GPU path stores
an intermediate in bf16 (the LoRA down-projection u, bf16 linear outputs, the bf16
activations of the Llama block), the oracle rounds at the same tensor boundary, so that
the two sides see the same storage format; all arithmetic between those boundaries is
fp64. Matrix products use numpy's matmul as a library primitive, with no blocking or
reordering of our own.

Paper references (section / algorithm / appendix of "Efficient RLHF: Reducing the Memory
Usage of PPO"):
  * §2 "Stage 3: PPO" -- LoRA on all linear layers; ratio and clipped surrogate; GAE uses
    V(x, y) to build the advantage estimates; critic trained on returns.
  * §3 "Dynamic LoRA" -- the reference policy is the actor with its LoRA parameters
    ignored, pi_ref <- LO(pi_theta); likewise the reward model is LO(critic).
  * §3 "Stage 2: Hydra-PPO" and Algorithm 1 (J-Hydra-PPO) / Algorithm 2 (Hydra-PPO) --
    one frozen base; the LoRA-off model supplies the reward and the reference
    log-probabilities, and the advantages are computed from them.
  * Appendix B "Experiment Details" -- KL coefficient beta = 0.02, GAE gamma = 1.0,
    lambda = 0.95, LoRA rank 128.

Readings where the paper is silent (the same readings the CUDA path implements):
  * LoRA update: y_on = x W + s (x A) B (Hu et al. 2021 form); s is an argument.
  * u = s * (x A) is stored in bf16 (the CUDA path keeps it as a bf16 operand).
  * Per-token KL penalty uses the sampled-token estimate logp_actor - logp_ref; the
    sequence score is added at the last valid token t = len - 1.
  * GAE: the value after the last valid token is 0 (terminal); positions >= len are 0.
  * Sampling: the paper does not say how tokens are drawn; temperature 1 sampling from the
    actor's softmax by the Gumbel-max trick, with the noise passed in (greedy without it).
  * PPO update side: the paper gives no clip range; eps = 0.2 (the PPO paper's default) is
    an argument. Losses are means over the valid tokens of the batch; the surrogate is
    negated so both losses are minimised. Advantage whitening (optional, off by default)
    uses the population variance over valid tokens with 1e-8 under the square root.

Parity pins for every function live in tests/test_oracle_pins.py (closed forms,
invariants, brute force, library routines, hand-worked fixtures in tests/golden/).
`set_storage_dither` (off by default) is a sensitivity probe used to derive the end-to-end
tolerance of the multi-layer composition; it never changes the default results.
The Llama composition (`llama_final_hidden` over `llama_layer`, under `llama_score` and the three-stream
Hydra-PPO pass `llama_score_hydra`) is pinned, with the bf16 storage rounding switched off,
against the same architecture built from PyTorch library operations in fp64 (F.linear,
F.rms_norm, causal F.scaled_dot_product_attention, F.silu, rotary as a complex rotation);
and through its per-op pieces and invariants (LoRA off, causality, one LoRA set reducing
Hydra-PPO to J-Hydra-PPO, a critic set that moves only the values). Where it rounds to bf16
(the tensors the GPU stores as bf16) is a reading, not pinned by that comparison.
Generation (`llama_generate`, the sampling phase of Alg. 1 and 2) recomputes
the whole stack at every step, with no cache, and draws each token by the Gumbel-max trick
from noise that is an input (`gumbel_argmax`, pinned by the empirical distribution of its
draws). It is pinned by its equality with `llama_score` on the finished sequence, and
through it by the library forward above.
"""
from __future__ import annotations

import numpy as np

# ---------------------------------------------------------------------------
# bf16 storage format (IEEE binary32 with the low 16 mantissa bits dropped)
# ---------------------------------------------------------------------------


def bf16_to_f64(bits) -> np.ndarray:
    """Widen bf16 bit patterns (uint16) to exact float64 values."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32).astype(np.float64)


def f64_to_bf16_bits(x) -> np.ndarray:
    """Round to bf16 (nearest, ties to even, via float32) and return uint16 bits."""
    f = np.ascontiguousarray(np.asarray(x, dtype=np.float64).astype(np.float32))
    u = f.view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    u = (u + np.uint64(0x7FFF) + lsb) >> np.uint64(16)
    return u.astype(np.uint16)


_DITHER = {"eps": 0.0, "rng": None}


def set_storage_dither(eps, seed=0):
    """Sensitivity probe (off by default): with eps > 0 every value is multiplied by
    (1 + eps * xi), xi = +-1 at random, before it is stored as bf16. A real fp32 kernel
    reaches each stored value through an accumulation order that differs from the exact
    fp64 sum by a relative amount of this size, so two dithered runs show how far equally
    valid roundings of the same chain drift apart. eps = 0 restores the plain oracle."""
    _DITHER["eps"] = float(eps)
    _DITHER["rng"] = np.random.default_rng(seed) if eps > 0 else None


def round_bf16(x) -> np.ndarray:
    """Value of x after storing it as bf16 (float64 result)."""
    if _DITHER["eps"] > 0:
        x = np.asarray(x, dtype=np.float64)
        xi = _DITHER["rng"].integers(0, 2, size=x.shape) * 2.0 - 1.0
        x = x * (1.0 + _DITHER["eps"] * xi)
    return bf16_to_f64(f64_to_bf16_bits(x))


# ---------------------------------------------------------------------------
# a1 / a2 / a3: dual-output LoRA linear (§2 Stage 3 LoRA; §3 Dynamic LoRA)
# Storage: x [M, K], W [N, K] (the paper's K x N weight, transposed), A [r, K], B [N, r].
# ---------------------------------------------------------------------------


def lora_down(x_on, A, s) -> np.ndarray:
    """u = s * (x_on A^T), stored as bf16. x_on, A: float64 arrays."""
    return round_bf16(s * (x_on @ A.T))


def dual_lora_linear(x_off, x_on, W, A, B, s, out_bf16=True):
    """(y_off, y_on) with y_off = x_off W^T (LoRA off, the reference / reward stream) and
    y_on = x_on W^T + u B^T with u = s x_on A^T (LoRA on, the actor / critic stream).

    §3 Dynamic LoRA: pi_ref <- LO(pi_theta), LO ignores the LoRA parameters, so the same
    frozen W produces both outputs. A is None means no LoRA on this linear (y_on = x_on W^T).
    """
    y_off = x_off @ W.T
    y_on = x_on @ W.T
    if A is not None:
        u = lora_down(x_on, A, s)
        y_on = y_on + u @ B.T
    if out_bf16:
        return round_bf16(y_off), round_bf16(y_on)
    return y_off, y_on


# ---------------------------------------------------------------------------
# a4: log-probability of the sampled token (Alg. 1/2: the LoRA-off model gives the reference
# log-probabilities; the §2 ratio r(theta) = pi_theta / pi_old needs the actor's too)
# ---------------------------------------------------------------------------


def logsumexp_rows(z) -> np.ndarray:
    """Textbook two-pass log-sum-exp per row: m = max_v z_v; m + log sum_v exp(z_v - m)."""
    m = np.max(z, axis=-1, keepdims=True)
    return (m + np.log(np.sum(np.exp(z - m), axis=-1, keepdims=True)))[..., 0]


def log_softmax_gather(z, ids):
    """(logp, lse): logp[t] = z[t, ids[t]] - lse[t], lse[t] = log sum_v exp(z[t, v])."""
    lse = logsumexp_rows(z)
    picked = np.take_along_axis(z, np.asarray(ids, dtype=np.int64)[:, None], axis=1)[:, 0]
    return picked - lse, lse


# ---------------------------------------------------------------------------
# a5: KL-penalised per-token reward (§2: a KL term against the reference policy keeps the
# actor near it; Appendix B KL coefficient beta; Alg. 1/2 reward from the LoRA-off model)
# ---------------------------------------------------------------------------


def kl_penalised_reward(logp_actor, logp_ref, lengths, score, beta):
    """r[s, t] = -beta (logp_actor - logp_ref) for t < len_s, plus score_s at t = len_s - 1;
    0 for t >= len_s. Inputs are [S, L] (score [S] or None)."""
    la = np.asarray(logp_actor, dtype=np.float64)
    lr = np.asarray(logp_ref, dtype=np.float64)
    S, L = la.shape
    t = np.arange(L)[None, :]
    n = np.asarray(lengths, dtype=np.int64)[:, None]
    valid = t < n
    r = np.where(valid, -beta * (la - lr), 0.0)
    if score is not None:
        last = (t == n - 1) & valid
        r = r + np.where(last, np.asarray(score, dtype=np.float64)[:, None], 0.0)
    return r


def token_logprobs_kl(z_actor, z_ref, ids, lengths, score, beta, S, L):
    """The hydra_token_logprobs_kl operation: z_* are [S*L, V] logit rows aligned with ids
    (row t predicts ids[t]); returns dict of [S, L] arrays (zero at t >= len) plus lse."""
    la, lse_a = log_softmax_gather(z_actor, ids)
    lr, lse_r = log_softmax_gather(z_ref, ids)
    la = la.reshape(S, L)
    lr = lr.reshape(S, L)
    if lengths is None:
        lengths = np.full(S, L, dtype=np.int64)
    valid = np.arange(L)[None, :] < np.asarray(lengths)[:, None]
    return {
        "logp_actor": np.where(valid, la, 0.0),
        "logp_ref": np.where(valid, lr, 0.0),
        "reward": kl_penalised_reward(la, lr, lengths, score, beta),
        "lse_actor": np.where(valid, lse_a.reshape(S, L), 0.0),
        "lse_ref": np.where(valid, lse_r.reshape(S, L), 0.0),
    }


# ---------------------------------------------------------------------------
# a7: generalised advantage estimation (§2: the advantage estimates come from GAE over the
# critic's values V(x, y), and the critic is trained on the returns; Appendix B gamma = 1.0,
# lambda = 0.95; Alg. 1/2 compute the advantages after scoring)
# ---------------------------------------------------------------------------


def gae(rewards, values, lengths, gamma, lam):
    """Plain backward recursion, one token at a time:
        delta_t = r_t + gamma * V_{t+1} - V_t      (V_{len} = 0: terminal)
        A_t     = delta_t + gamma * lam * A_{t+1}  (A_{len} = 0)
        R_t     = A_t + V_t
    Positions t >= len are 0 in both outputs."""
    r = np.asarray(rewards, dtype=np.float64)
    v = np.asarray(values, dtype=np.float64)
    S, L = r.shape
    adv = np.zeros((S, L))
    ret = np.zeros((S, L))
    for s in range(S):
        n = int(lengths[s]) if lengths is not None else L
        a_next = 0.0
        for t in range(n - 1, -1, -1):
            v_next = v[s, t + 1] if t + 1 < n else 0.0
            delta = r[s, t] + gamma * v_next - v[s, t]
            a = delta + gamma * lam * a_next
            adv[s, t] = a
            ret[s, t] = a + v[s, t]
            a_next = a
    return adv, ret


# ---------------------------------------------------------------------------
# a8: Llama decoder pieces used by the full scoring pass (the paper uses Llama 7b, §4)
# ---------------------------------------------------------------------------


def rmsnorm(h, w, eps):
    """RMSNorm (Zhang & Sennrich 2019): h / sqrt(mean(h^2) + eps) * w, per row."""
    h = np.asarray(h, dtype=np.float64)
    return h / np.sqrt(np.mean(h * h, axis=-1, keepdims=True) + eps) * w


def rope(x, positions, theta):
    """Rotary embedding (Su et al. 2021), rotate-half pairing: dims (i, i + D/2) of each
    head form one plane rotated by angle pos * theta^(-2i/D). x: [T, H, D]."""
    T, H, D = x.shape
    half = D // 2
    inv = theta ** (-np.arange(half, dtype=np.float64) * 2.0 / D)
    ang = np.asarray(positions, dtype=np.float64)[:, None] * inv[None, :]  # [T, half]
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    x1 = x[..., :half]
    x2 = x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x1 * s + x2 * c], axis=-1)


def causal_attention(q, k, v):
    """softmax(q k^T / sqrt(D) + causal mask) v per head. q, k, v: [T, H, D] -> [T, H, D]."""
    T, H, D = q.shape
    out = np.empty((T, H, D))
    mask = np.triu(np.ones((T, T), dtype=bool), 1)
    for h in range(H):
        sc = (q[:, h, :] @ k[:, h, :].T) / np.sqrt(D)
        sc = np.where(mask, -np.inf, sc)
        m = np.max(sc, axis=1, keepdims=True)
        p = np.exp(sc - m)
        p = p / np.sum(p, axis=1, keepdims=True)
        out[:, h, :] = p @ v[:, h, :]
    return out


def silu(x):
    return x / (1.0 + np.exp(-x))


def swiglu(g, u):
    """SwiGLU gate (Shazeer 2020): silu(g) * u."""
    return silu(g) * u


def llama_layer(weights, l, h_off, h_on, cfg):
    """Decoder layer l of both streams (LoRA off / on, §3 Dynamic LoRA) on the residual
    streams h_off, h_on [T, d] of one sequence (positions 0..T-1): pre-norm attention with
    the rotary embedding, then the pre-norm SwiGLU feed-forward, each added into the residual
    stream. Returns the new (h_off, h_on)."""
    d = cfg["d"]
    H = cfg["n_heads"]
    Dh = d // H
    eps = cfg["eps"]
    s = cfg["lora_scale"]
    T = h_off.shape[0]
    pos = np.arange(T)

    def lin(name, a_off, a_on):
        W = weights[name][l]
        ab = weights["lora"].get(name)
        if ab is None:
            return dual_lora_linear(a_off, a_on, W, None, None, s)
        return dual_lora_linear(a_off, a_on, W, ab[0][l], ab[1][l], s)

    a_off = round_bf16(rmsnorm(h_off, weights["norm1"][l], eps))
    a_on = round_bf16(rmsnorm(h_on, weights["norm1"][l], eps))
    q = lin("wq", a_off, a_on)
    k = lin("wk", a_off, a_on)
    v = lin("wv", a_off, a_on)
    att = []
    for i in range(2):
        qi = round_bf16(rope(q[i].reshape(T, H, Dh), pos, cfg["rope_theta"]))
        ki = round_bf16(rope(k[i].reshape(T, H, Dh), pos, cfg["rope_theta"]))
        vi = v[i].reshape(T, H, Dh)
        att.append(round_bf16(causal_attention(qi, ki, vi).reshape(T, d)))
    o = lin("wo", att[0], att[1])
    h_off = h_off + o[0]
    h_on = h_on + o[1]
    a_off = round_bf16(rmsnorm(h_off, weights["norm2"][l], eps))
    a_on = round_bf16(rmsnorm(h_on, weights["norm2"][l], eps))
    g = lin("wg", a_off, a_on)
    u = lin("wu", a_off, a_on)
    m_off = round_bf16(swiglu(g[0], u[0]))
    m_on = round_bf16(swiglu(g[1], u[1]))
    dn = lin("wd", m_off, m_on)
    return h_off + dn[0], h_on + dn[1]


def llama_final_hidden(weights, ids, cfg, n_layers=None):
    """Final normed hidden states (bf16 values) of both streams at every position of one
    sequence: the decoder stack of the J-Hydra model (LoRA off / on, §3 Dynamic LoRA), as
    used by llama_score; row p is the state after token p, which predicts token p + 1."""
    eps = cfg["eps"]
    n_layers = cfg["n_layers"] if n_layers is None else n_layers
    h_off = weights["embed"][np.asarray(ids)]
    h_on = h_off.copy()
    for l in range(n_layers):
        h_off, h_on = llama_layer(weights, l, h_off, h_on, cfg)
    f_off = round_bf16(rmsnorm(h_off, weights["final_norm"], eps))
    f_on = round_bf16(rmsnorm(h_on, weights["final_norm"], eps))
    return f_off, f_on


def llama_score(weights, ids, prompt_len, cfg, seq_lengths=None, beta=0.1, gamma=1.0,
                lam=0.95, n_layers=None):
    """One sequence of the full J-Hydra scoring pass (Alg. 1 scoring steps), both streams.

    weights: dict of float64 arrays (exact bf16 values):
      embed [V, d]; per layer l: wq, wk, wv, wo [d, d]; wg, wu [F, d]; wd [d, F];
      norm1, norm2 [d]; lora[name] = (A [r, in], B [out, r]) for name in q, v, g, u, d;
      final_norm [d]; lm_head [V, d]; w_rm [d].
    ids: [T] token ids (prompt then response); prompt_len P; response tokens are P..T-1.
    Returns dict with logp_actor, logp_ref, reward, values, score, advantages, returns
    (arrays of length T-P for the response) and the final normed hidden states.

    Streams: "off" = LoRA ignored (reference policy and reward model, §3 Dynamic LoRA);
    "on" = actor/critic with the single J-Hydra LoRA set (§3 J-Hydra-PPO).
    Values: V_t = w_rm . h_on[p_t - 1]; score = w_rm . h_off[T - 1] (reward-model head on
    the LoRA-off stream, critic = same head with LoRA on).
    """
    P = prompt_len
    T = len(ids)
    L = T - P
    f_off, f_on = llama_final_hidden(weights, ids, cfg, n_layers)
    rows = np.arange(P - 1, T - 1)                       # hidden row predicting token P+t
    z_ref = f_off[rows] @ weights["lm_head"].T
    z_act = f_on[rows] @ weights["lm_head"].T
    resp_ids = np.asarray(ids)[P:]
    la, _ = log_softmax_gather(z_act, resp_ids)
    lr, _ = log_softmax_gather(z_ref, resp_ids)
    n = L if seq_lengths is None else int(seq_lengths)
    score = float(f_off[P - 1 + n] @ weights["w_rm"]) if n > 0 else 0.0
    values = f_on[rows] @ weights["w_rm"]
    reward = kl_penalised_reward(la[None], lr[None], [n], [score], beta)[0]
    adv, ret = gae(reward[None], values[None], [n], gamma, lam)
    valid = np.arange(L) < n
    return {
        "logp_actor": np.where(valid, la, 0.0),
        "logp_ref": np.where(valid, lr, 0.0),
        "reward": reward,
        "values": np.where(valid, values, 0.0),
        "score": score,
        "advantages": adv[0],
        "returns": ret[0],
        "h_off": f_off,
        "h_on": f_on,
    }


def llama_score_hydra(weights, lora_critic, ids, prompt_len, cfg, seq_lengths=None, beta=0.1,
                      gamma=1.0, lam=0.95, n_layers=None):
    """One sequence of the Hydra-PPO scoring pass (Alg. 2 scoring steps): three streams of
    the same frozen base model (§3 Stage 2: two LoRA sets on one base; dynamic LoRA):
      off    LoRA ignored: reference log-probabilities and the reward score,
      actor  the actor's LoRA set weights["lora"]: the policy log-probabilities,
      critic the critic's LoRA set lora_critic: the values through the reward head,
             r_phi <- LO(V), so V_t = w_rm . h_critic[p_t - 1].
    weights, ids, prompt_len, cfg as llama_score; lora_critic has the layout of
    weights["lora"]. Returns llama_score's outputs with values from the critic stream and
    the final normed hidden states h_off, h_act, h_crit. With lora_critic equal to the
    actor's set this is J-Hydra-PPO and the outputs equal llama_score's."""
    d = cfg["d"]
    H = cfg["n_heads"]
    Dh = d // H
    eps = cfg["eps"]
    s = cfg["lora_scale"]
    T = len(ids)
    P = prompt_len
    L = T - P
    n_layers = cfg["n_layers"] if n_layers is None else n_layers
    pos = np.arange(T)
    sets = [None, weights["lora"], lora_critic]

    def lin1(name, l, a, lora):
        # one stream of the dual-output linear: no LoRA, or this stream's LoRA set
        W = weights[name][l]
        ab = None if lora is None else lora.get(name)
        if ab is None:
            return dual_lora_linear(a, a, W, None, None, s)[0]
        return dual_lora_linear(a, a, W, ab[0][l], ab[1][l], s)[1]

    h = [weights["embed"][np.asarray(ids)] for _ in range(3)]
    for l in range(n_layers):
        for i, lora in enumerate(sets):
            a = round_bf16(rmsnorm(h[i], weights["norm1"][l], eps))
            q = lin1("wq", l, a, lora)
            k = lin1("wk", l, a, lora)
            v = lin1("wv", l, a, lora)
            qi = round_bf16(rope(q.reshape(T, H, Dh), pos, cfg["rope_theta"]))
            ki = round_bf16(rope(k.reshape(T, H, Dh), pos, cfg["rope_theta"]))
            att = round_bf16(causal_attention(qi, ki, v.reshape(T, H, Dh)).reshape(T, d))
            h[i] = h[i] + lin1("wo", l, att, lora)
            a = round_bf16(rmsnorm(h[i], weights["norm2"][l], eps))
            m = round_bf16(swiglu(lin1("wg", l, a, lora), lin1("wu", l, a, lora)))
            h[i] = h[i] + lin1("wd", l, m, lora)

    f = [round_bf16(rmsnorm(hi, weights["final_norm"], eps)) for hi in h]
    rows = np.arange(P - 1, T - 1)                       # hidden row predicting token P+t
    resp_ids = np.asarray(ids)[P:]
    lr, _ = log_softmax_gather(f[0][rows] @ weights["lm_head"].T, resp_ids)
    la, _ = log_softmax_gather(f[1][rows] @ weights["lm_head"].T, resp_ids)
    n = L if seq_lengths is None else int(seq_lengths)
    score = float(f[0][P - 1 + n] @ weights["w_rm"]) if n > 0 else 0.0
    values = f[2][rows] @ weights["w_rm"]
    reward = kl_penalised_reward(la[None], lr[None], [n], [score], beta)[0]
    adv, ret = gae(reward[None], values[None], [n], gamma, lam)
    valid = np.arange(L) < n
    return {
        "logp_actor": np.where(valid, la, 0.0),
        "logp_ref": np.where(valid, lr, 0.0),
        "reward": reward,
        "values": np.where(valid, values, 0.0),
        "score": score,
        "advantages": adv[0],
        "returns": ret[0],
        "h_off": f[0],
        "h_act": f[1],
        "h_crit": f[2],
    }


# ---------------------------------------------------------------------------
# Update side of PPO (§2 Stage 3: ratio r(theta), clipped surrogate L^CLIP, squared-error
# value loss on the returns; Alg. 1/2 optimise this surrogate after each batch is scored)
# ---------------------------------------------------------------------------


def ppo_loss(logp_new, logp_old, adv, returns, values, lengths, clip_eps=0.2, whiten=False,
             moments=None):
    """PPO losses over the valid tokens t < len_s of [S, L] arrays:
      r_t       = exp(logp_new_t - logp_old_t)                         (probability ratio)
      A_t       = adv_t, or (adv_t - mean) / sqrt(M2 / n + 1e-8) if whiten
      s_t       = min(r_t A_t, clip(r_t, 1 - eps, 1 + eps) A_t)
      loss_clip = -(1/n) sum_t s_t                                     (maximise L^CLIP)
      loss_value = (1/n) sum_t (values_t - returns_t)^2
    (n, mean, M2) are the count, mean and summed squared deviation of the valid advantages,
    or the given `moments` (e.g. those of a larger batch this one is a shard of; n then
    also normalises the losses).
    Returns dict with loss_clip, loss_value, clip_frac (share of valid tokens with
    |r - 1| > eps, over n), approx_kl ((1/n) sum (logp_old - logp_new)), adv_mean, adv_std
    (mean and population std of the raw advantages: from `moments` when given, else of
    this batch), n, grad_logp = d loss_clip / d logp_new and grad_values =
    d loss_value / d values (0 at invalid tokens). A_t is treated as a constant; where the
    two surrogate terms tie, the unclipped one carries the gradient."""
    ln = np.asarray(logp_new, dtype=np.float64)
    lo = np.asarray(logp_old, dtype=np.float64)
    a = np.asarray(adv, dtype=np.float64)
    R = np.asarray(returns, dtype=np.float64)
    V = np.asarray(values, dtype=np.float64)
    S, L = ln.shape
    valid = np.arange(L)[None, :] < np.asarray(lengths, dtype=np.int64).reshape(S, 1)
    if moments is None:
        n = float(valid.sum())
        mean = float(a[valid].sum() / n) if n > 0 else 0.0
        m2 = float(((a[valid] - mean) ** 2).sum())
    else:
        n, mean, m2 = (float(v) for v in moments)
    var = m2 / n if n > 0 else 0.0
    inv_n = 1.0 / n if n > 0 else 0.0
    A = (a - mean) / np.sqrt(var + 1e-8) if whiten else a
    r = np.exp(ln - lo)
    rc = np.clip(r, 1.0 - clip_eps, 1.0 + clip_eps)
    unclipped, clip_term = r * A, rc * A
    surr = np.minimum(unclipped, clip_term)
    dv = V - R
    return {
        "loss_clip": -float(surr[valid].sum()) * inv_n,
        "loss_value": float((dv[valid] ** 2).sum()) * inv_n,
        "clip_frac": float((valid & (np.abs(r - 1.0) > clip_eps)).sum()) * inv_n,
        "approx_kl": float((lo - ln)[valid].sum()) * inv_n,
        "adv_mean": mean,
        "adv_std": float(np.sqrt(var)),
        "n": n,
        "grad_logp": np.where(valid & (unclipped <= clip_term), -unclipped * inv_n, 0.0),
        "grad_values": np.where(valid, 2.0 * dv * inv_n, 0.0),
    }


# ---------------------------------------------------------------------------
# Generation with the actor (Alg. 1 and 2: the actor samples each sequence for T steps;
# J-Hydra-PPO keeps the critic head's values while sampling)
# ---------------------------------------------------------------------------


def gumbel_argmax(z, g=None):
    """One draw from softmax(z) by the Gumbel-max trick (Gumbel 1954; Maddison, Tarlow and
    Minka 2014): argmax_k (z_k + g_k) with g_k i.i.d. standard Gumbel (-log(-log U)). The
    noise is an input; g None is the greedy argmax. Ties go to the lowest index."""
    z = np.asarray(z, dtype=np.float64)
    return int(np.argmax(z if g is None else z + np.asarray(g, dtype=np.float64)))


def llama_generate(weights, prompt_ids, n_steps, cfg, gumbel=None, n_layers=None):
    """Autoregressive generation of n_steps tokens after the prompt with the LoRA-on actor,
    recording under both streams the log-probability of each drawn token and the J-Hydra
    value of the state it is drawn from. No cache: step t runs the whole decoder stack over
    the prompt and the t tokens drawn so far (the plain definition of a causal model's
    next-token distribution) and reads the last position p = P0 + t - 1:
      z_on = lm_head f_on[p], z_off = lm_head f_off[p]
      token_t      = argmax_k (z_on[k] + gumbel[t, k])   (greedy when gumbel is None)
      logp_actor_t = log_softmax(z_on)[token_t],  logp_ref_t = log_softmax(z_off)[token_t]
      value_t      = w_rm . f_on[p]
    score = w_rm . f_off at the last drawn token (one more pass over the whole sequence).
    These are llama_score's logp_actor, logp_ref, values and score on the generated
    sequence. gumbel: [n_steps, V] or None. Returns a dict of tokens (int array),
    logp_actor, logp_ref, values (length n_steps) and score."""
    ids = [int(t) for t in prompt_ids]
    P = len(ids)
    out = {k: np.zeros(n_steps) for k in ("logp_actor", "logp_ref", "values")}
    tokens = np.zeros(n_steps, dtype=np.int64)
    for t in range(n_steps):
        f_off, f_on = llama_final_hidden(weights, ids, cfg, n_layers)
        z_on = f_on[-1] @ weights["lm_head"].T
        z_off = f_off[-1] @ weights["lm_head"].T
        tok = gumbel_argmax(z_on, None if gumbel is None else gumbel[t])
        out["logp_actor"][t] = z_on[tok] - logsumexp_rows(z_on[None])[0]
        out["logp_ref"][t] = z_off[tok] - logsumexp_rows(z_off[None])[0]
        out["values"][t] = float(f_on[-1] @ weights["w_rm"])
        tokens[t] = tok
        ids.append(tok)
    f_off, _ = llama_final_hidden(weights, ids, cfg, n_layers)
    out["score"] = float(f_off[-1] @ weights["w_rm"])
    out["tokens"] = tokens
    out["prompt_len"] = P
    return out
