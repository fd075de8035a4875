/*
 * libhydra: GB300 (sm_103a) kernels for the experience-scoring step of Hydra-PPO
 * ("Efficient RLHF: Reducing the Memory Usage of PPO", arXiv 2309.00754).
 *
 * In Hydra-PPO a single frozen base model plays several roles. With its LoRA parameters
 * ignored it is the reference policy (and, in J-Hydra-PPO, the reward model); with LoRA
 * switched on it is the actor (§3 "Dynamic LoRA": pi_ref <- LO(pi_theta); §3 "Stage 2:
 * Hydra-PPO"; Algorithm 1 and 2). Scoring a generated batch therefore needs, per frozen
 * weight W, both the LoRA-off and the LoRA-on output, then the log-probability of every
 * sampled token under both heads, a KL-penalised per-token reward, and generalised
 * advantage estimates (§2 "Stage 3: PPO"; Appendix B: beta, gamma, lambda).
 *
 * Conventions shared by every entry point:
 *  - All tensor pointers are DEVICE pointers owned by the caller; the library never frees
 *    them and keeps no reference after the call returns. The library allocates no device
 *    memory per call; scratch space, where needed, is a caller-provided workspace.
 *  - Matrices are row-major and dense (row stride = number of columns) unless a leading
 *    dimension argument says otherwise. "bf16" is IEEE binary32 with the low 16 mantissa
 *    bits removed; accumulation is fp32.
 *  - `stream` is a cudaStream_t passed as void* (NULL = the legacy default stream). Every
 *    call is asynchronous on that stream; nothing synchronises except
 *    hydra_device_error().
 *  - Argument errors are detected on the host and returned before anything is launched.
 *    Errors found by a kernel (a token id outside [0, V), a length outside [0, L], a
 *    bounded wait that ran out) are recorded in the library's device error word (first
 *    error wins) and read with hydra_device_error(); the affected outputs hold NaN. No
 *    kernel traps.
 *  - Outputs must not alias inputs (x_on == x_off is the one meaningful alias).
 */
#ifndef HYDRA_H_
#define HYDRA_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum hydra_status {
  HYDRA_OK = 0,
  HYDRA_ERR_NULL = 1,      /* a required pointer is NULL */
  HYDRA_ERR_SHAPE = 2,     /* a size is negative or outside the supported range */
  HYDRA_ERR_ALIGN = 3,     /* a pointer or row length breaks the 16-byte rule */
  HYDRA_ERR_RANGE = 4,     /* a scalar or enum argument is out of range */
  HYDRA_ERR_CUDA = 5,      /* a CUDA runtime/driver call failed (launch, tensor map) */
  HYDRA_ERR_TIMEOUT = 6,   /* device error word: a bounded in-kernel wait expired */
  HYDRA_ERR_WORKSPACE = 7, /* workspace missing or smaller than the query says */
  HYDRA_ERR_DEVICE = 8     /* device error word: bad token id or sequence length */
} hydra_status;

typedef enum hydra_dtype { HYDRA_BF16 = 0, HYDRA_F32 = 1 } hydra_dtype;

/* Static, human-readable name of a status code. */
const char* hydra_status_string(int status);

/* ABI version of this header (incremented on any signature change). */
int hydra_abi_version(void);

/*
 * Read (and optionally clear) the device error word of the current CUDA device.
 * Synchronises the device. *code_out receives 0 when no kernel has reported an error,
 * otherwise the first code recorded (0x1xx: bounded wait expired, 0x201: token id out of
 * range, 0x202: sequence length out of range). Returns HYDRA_OK, HYDRA_ERR_NULL or
 * HYDRA_ERR_CUDA.
 */
hydra_status hydra_device_error(int32_t* code_out, int clear);

/*
 * Self-test of the in-kernel failure detection: one CTA waits on an mbarrier that nothing
 * ever signals, through the same bounded wait every kernel of the library uses. The wait
 * expires after about 2e9 SM clock cycles (about 1 s), the kernel records 0x105 in the
 * device error word and returns; nothing traps and the context stays usable. Asynchronous
 * on `stream` (a cudaStream_t, NULL = default); read the code with hydra_device_error.
 * Returns HYDRA_OK, or HYDRA_ERR_CUDA when the launch fails.
 */
hydra_status hydra_selftest_wait_timeout(void* stream);

/*
 * LoRA down-projection (§2 Stage 3: LoRA on all linear layers; the update is
 * y = x W + s (x A) B): u = s * (x_on A^T), rounded to bf16.
 *   x_on : bf16 [M, K]       A : bf16 [r, K] (the paper's K x r matrix A, transposed)
 *   u    : bf16 [M, r] (output)
 * K % 8 == 0, 1 <= r <= 256, r % 8 == 0, pointers 16-byte aligned. M == 0 is a no-op.
 */
hydra_status hydra_lora_down(const void* x_on, int64_t M, int64_t K, const void* A, int64_t r,
                             float s, void* u, void* stream);

/* Bytes of workspace hydra_lora_linear needs for M token rows and rank r (0 when r == 0). */
size_t hydra_lora_linear_workspace_size(int64_t M, int64_t r);

/*
 * Dual-output LoRA linear: one pass over the frozen weight W yields the LoRA-off and the
 * LoRA-on output (§3 Dynamic LoRA, pi_ref <- LO(pi_theta); §2 Stage 3 LoRA update):
 *     y_off = x_off W^T
 *     y_on  = x_on  W^T + u B^T,   u = s (x_on A^T) stored as bf16
 * Arguments:
 *   x_off : bf16 [M, K] input of the LoRA-off stream (reference / reward model).
 *   x_on  : bf16 [M, K] input of the LoRA-on stream (actor / critic). Pass x_on == x_off
 *           (or NULL) when both streams share the input: W x is then accumulated once and
 *           both outputs leave the same tensor-core accumulator.
 *   W     : bf16 [N, K], nn.Linear layout (the paper's K x N weight, transposed).
 *   A, B  : bf16 [r, K] and [N, r]; r == 0 (A, B ignored) means no LoRA on this linear,
 *           so y_on = x_on W^T. Otherwise 8 <= r <= 256 and r % 8 == 0.
 *   s     : LoRA scale (the paper does not fix it; alpha / r in the usual notation).
 *   y_off, y_on : [M, N] outputs of dtype out_dtype (HYDRA_BF16 or HYDRA_F32), either may
 *           be NULL (not both).
 *   workspace : device scratch of at least hydra_lora_linear_workspace_size(M, r) bytes,
 *           16-byte aligned; holds u between the two kernels of the call. It may be
 *           reused as soon as the call's work on `stream` has completed.
 * Requirements: K % 8 == 0 and N % 8 == 0 (16-byte rows), all pointers 16-byte aligned,
 * M, N, K < 2^31. M == 0 is a no-op. Up to 16 token rows over both streams take the
 * memory-bound GEMV kernel; larger M the tcgen05 tensor-core kernel.
 */
hydra_status hydra_lora_linear(const void* x_off, const void* x_on, int64_t M, int64_t K,
                               int64_t N, const void* W, const void* A, const void* B, int64_t r,
                               float s, void* y_off, void* y_on, int out_dtype, void* workspace,
                               size_t workspace_bytes, void* stream);

/*
 * The dual-output linear given a precomputed LoRA down-projection u (the second half of
 * hydra_lora_linear, for callers that keep u, e.g. to time the two kernels apart):
 *     y_off = x_off W^T,   y_on = x_on W^T + u B^T
 *   u : bf16 [M, r] = s (x_on A^T) as written by hydra_lora_down; B : bf16 [N, r].
 *   r == 0 (u, B ignored) means no LoRA. algo: 0 automatic, 1 tcgen05 tile kernel,
 *   2 GEMV (at most 16 token rows over both streams), 3 tcgen05 single-CTA tiles.
 * Same layout, alignment and error rules as hydra_lora_linear; no workspace.
 */
hydra_status hydra_dual_linear(const void* x_off, const void* x_on, int64_t M, int64_t K,
                               int64_t N, const void* W, const void* u, const void* B, int64_t r,
                               void* y_off, void* y_on, int out_dtype, int algo, void* stream);

/*
 * The decode-step form of hydra_dual_linear (§3 Dynamic LoRA: one frozen W serves both
 * streams): the two streams' token rows stacked in one matrix x = [x_off; x_on], at most
 * 128 rows, and
 *     y[i] = x[i] W^T                          for every row i in [0, M)
 *     y[i] = x[i] W^T + u[i - u_row0] B^T      for i in [u_row0, u_row0 + u_rows)
 * on a tcgen05 kernel that splits K over a thread-block cluster, so that a weight read
 * once, by only a few output tiles, still streams through most of the device's SMs.
 *   x : bf16 [M, K], 0 <= M <= 128 (M == 0 is a no-op).   W : bf16 [N, K].
 *   y : [M, N] of out_dtype (HYDRA_BF16: the fp32 sum rounded once; HYDRA_F32).
 *   u : bf16 [u_rows, r] (s x_on A^T, as hydra_lora_down writes it); B : bf16 [N, r].
 *       r == 0 means no LoRA (u, B, u_row0, u_rows ignored); otherwise 8 <= r <= 256,
 *       r % 8 == 0, u_rows >= 1, u_row0 >= 0 and u_row0 + u_rows <= M.
 *   tile_n  : output tile width, a multiple of 16 up to 256; 0 = chosen by the library.
 *   split_k : CTAs of a cluster splitting K, 1..8 and at most ceil(K / 64); 0 = chosen.
 *       The partial sums are added in a fixed order, so a given (tile_n, split_k) gives
 *       the same bits on every call; different choices associate the fp32 sums
 *       differently.
 * Requirements: K % 8 == 0, N % 16 == 0, all pointers 16-byte aligned, K, N < 2^31.
 * Errors: HYDRA_ERR_NULL (x, W or y NULL; u or B NULL with r > 0), HYDRA_ERR_SHAPE (M, N,
 * r, u_row0 or u_rows out of range), HYDRA_ERR_ALIGN (misaligned pointer, K % 8 != 0,
 * r % 8 != 0), HYDRA_ERR_RANGE (out_dtype, tile_n or split_k), HYDRA_ERR_CUDA (launch).
 */
hydra_status hydra_skinny_linear(const void* x, int64_t M, int64_t K, int64_t N, const void* W,
                                 const void* u, int64_t u_row0, int64_t u_rows, const void* B,
                                 int64_t r, void* y, int out_dtype, int tile_n, int split_k,
                                 void* stream);

/*
 * Hydra-PPO's three streams through one frozen weight (Algorithm 2: the critic LoRA gives
 * the values, LoRA off the reward and reference log-probabilities, the actor LoRA the policy;
 * §3 Stage 2: two LoRA sets on one base model):
 *     y_off  = x_off  W^T
 *     y_act  = x_act  W^T + u_a B_act^T,    u_a = s (x_act  A_act^T)  stored as bf16
 *     y_crit = x_crit W^T + u_c B_crit^T,   u_c = s (x_crit A_crit^T) stored as bf16
 * on the tcgen05 kernel with the three streams' tiles of one output block adjacent, so each W
 * tile comes from HBM once and twice more from L2. Inputs may alias one another (the first
 * layer of a pass); any output may be NULL (not all three), and a NULL output's LoRA set may
 * be NULL. With A_crit = A_act, B_crit = B_act and x_crit = x_act, y_crit equals y_act bit
 * for bit (J-Hydra's single LoRA set). Layouts, alignment and errors as hydra_lora_linear;
 * workspace: hydra_lora_linear_tri_workspace_size(M, r) bytes (both u).
 */
size_t hydra_lora_linear_tri_workspace_size(int64_t M, int64_t r);
hydra_status hydra_lora_linear_tri(const void* x_off, const void* x_act, const void* x_crit,
                                   int64_t M, int64_t K, int64_t N, const void* W,
                                   const void* A_act, const void* B_act, const void* A_crit,
                                   const void* B_crit, int64_t r, float s, void* y_off,
                                   void* y_act, void* y_crit, int out_dtype, void* workspace,
                                   size_t workspace_bytes, void* stream);

/* Epilogues of hydra_dual_linear_ex. */
enum {
  HYDRA_EPI_STORE = 0,    /* y = result (bf16 or fp32), as hydra_dual_linear */
  HYDRA_EPI_SWIGLU = 1,   /* gated FFN: see hydra_dual_linear_ex */
  HYDRA_EPI_RESIDUAL = 2  /* residual stream update: see hydra_dual_linear_ex */
};

/*
 * hydra_dual_linear on the tcgen05 kernel with a fused epilogue (Llama decoder blocks of the
 * scoring pass; §4 uses Llama 7b):
 *  HYDRA_EPI_STORE    as hydra_dual_linear (algo 1).
 *  HYDRA_EPI_SWIGLU   W rows come in blocks of 128: block 2j holds gate rows, block 2j + 1 the
 *                     up rows of the same 128 features (B rows likewise; N % 256 == 0).
 *                     y_* are bf16 [M, N/2]: y[:, 128 j + i] = bf16(silu(g) * u) with
 *                     g = bf16(gate row 256 j + i), u = bf16(up row 256 j + 128 + i),
 *                     silu(g) = g / (1 + exp(-g)) (Shazeer 2020).
 *  HYDRA_EPI_RESIDUAL y_* are fp32 [M, N] residual streams, updated in place:
 *                     y += float(bf16(x W^T (+ u B^T))). Outputs of different calls may not
 *                     overlap in flight; within one call every element is updated once.
 * out_dtype applies to HYDRA_EPI_STORE only. Other arguments and errors as hydra_dual_linear.
 */
hydra_status hydra_dual_linear_ex(const void* x_off, const void* x_on, int64_t M, int64_t K,
                                  int64_t N, const void* W, const void* u, const void* B,
                                  int64_t r, void* y_off, void* y_on, int out_dtype, int epilogue,
                                  void* stream);

/*
 * Rotation table of the rotary position embedding (RoFormer, rotate-half pairing, as used by
 * hydra_rope): table[2 (pos * head_dim/2 + i) + {0, 1}] = (cos a, sin a) with
 * a = pos * theta^(-2i/head_dim), evaluated in fp32 exactly as hydra_rope evaluates it, for
 * pos in [0, P) and pair i in [0, head_dim/2). table: fp32 [P, head_dim/2, 2], 16-byte
 * aligned, caller-owned. Errors: NULL table -> HYDRA_ERR_NULL; P < 0, odd or < 2 head_dim ->
 * HYDRA_ERR_SHAPE; theta <= 0 -> HYDRA_ERR_RANGE; misaligned table -> HYDRA_ERR_ALIGN.
 */
hydra_status hydra_rope_table(int64_t P, int64_t head_dim, float theta, float* table,
                              void* stream);

/*
 * hydra_dual_linear on the tcgen05 kernel with the rotary position embedding of the Llama
 * attention fused into the epilogue, for the fused q/k/v projection: every output value is
 * first rounded to bf16 (the value hydra_dual_linear would store); then on columns
 * [0, rope_cols), in heads of head_dim = 128, the pairs (i, i + 64) of a head become
 *     x_i cos(a) - x_{i+64} sin(a),   x_i sin(a) + x_{i+64} cos(a)
 * with (cos a, sin a) = rope_table[row % P][i] (hydra_rope_table with this P and head_dim;
 * rows of each stream are sequences of P tokens), each product and sum rounded as hydra_rope
 * rounds them, so the result equals hydra_dual_linear followed by hydra_rope bit for bit.
 * Columns from rope_cols on are stored as hydra_dual_linear would. bf16 outputs only.
 * Errors: as hydra_dual_linear_ex; NULL rope_table -> HYDRA_ERR_NULL; misaligned
 * rope_table -> HYDRA_ERR_ALIGN; head_dim != 128 -> HYDRA_ERR_RANGE; P < 1,
 * rope_cols % 128 != 0 or rope_cols > N -> HYDRA_ERR_SHAPE.
 */
hydra_status hydra_dual_linear_rope(const void* x_off, const void* x_on, int64_t M, int64_t K,
                                    int64_t N, const void* W, const void* u, const void* B,
                                    int64_t r, void* y_off, void* y_on, int64_t P,
                                    int64_t rope_cols, int64_t head_dim, const float* rope_table,
                                    void* stream);

/*
 * hydra_lora_linear with the kernel family chosen by the caller:
 *   algo 0 = automatic (as hydra_lora_linear), 1 = tcgen05 tile kernel (any M; CTA pairs
 *   with 256-row tiles when M > 128), 2 = GEMV kernel (requires at most 16 token rows over
 *   both streams), 3 = tcgen05 tile kernel on single CTAs only (128-row tiles).
 * Same arguments, results and errors otherwise; algo outside 0..3 is HYDRA_ERR_RANGE.
 */
hydra_status hydra_lora_linear_algo(const void* x_off, const void* x_on, int64_t M, int64_t K,
                                    int64_t N, const void* W, const void* A, const void* B,
                                    int64_t r, float s, void* y_off, void* y_on, int out_dtype,
                                    void* workspace, size_t workspace_bytes, int algo,
                                    void* stream);

/* Largest M * r that hydra_lora_linear_noalloc accepts (u elements, bf16: 4 MiB). */
#define HYDRA_NOALLOC_MAX_U_ELEMS (1 << 21)

/*
 * hydra_lora_linear for callers that cannot allocate device memory: a plugin inside a
 * host framework that owns the device memory pool and passes it only its input and output
 * buffers, or a latency-critical caller that cannot afford cudaMalloc/cudaFree (they may
 * synchronise the device). The paper has no counterpart to this entry point.
 * Same arguments, results and argument errors as hydra_lora_linear, without the workspace:
 * u = s x_on A^T lives in a static device array of HYDRA_NOALLOC_MAX_U_ELEMS bf16 elements
 * (4 MiB) that every device which loads the library holds until the process exits; the
 * call allocates nothing.
 *  - M * r > HYDRA_NOALLOC_MAX_U_ELEMS (with LoRA active) returns HYDRA_ERR_SHAPE and
 *    launches nothing.
 *  - The first call on a device resolves the array's address on that device (device set-up);
 *    make it before any stream capture on that device.
 *  - All calls share the array. Calls whose work overlaps on the GPU (different streams, or
 *    unordered host threads) race on it; serialise them, e.g. on one stream.
 */
hydra_status hydra_lora_linear_noalloc(const void* x_off, const void* x_on, int64_t M, int64_t K,
                                       int64_t N, const void* W, const void* A, const void* B,
                                       int64_t r, float s, void* y_off, void* y_on, int out_dtype,
                                       void* stream);

/*
 * Per-token log-probabilities of the sampled tokens under the actor (LoRA on) and the
 * reference (LoRA off) heads, and the KL-penalised reward (Algorithm 1/2: LoRA off gives
 * the reference log-probabilities and the reward, which feed the advantage estimate;
 * §2: the reference keeps the policy from diverging; Appendix B: KL coefficient beta):
 *     lse_h[t]    = log sum_v exp z_h[t, v]
 *     logp_h[t]   = z_h[t, ids[t]] - lse_h[t]                    (h = actor, ref)
 *     reward[t]   = -beta (logp_actor[t] - logp_ref[t]) + [t == len_s - 1] seq_score[s]
 * Arguments:
 *   logits_actor, logits_ref : [S*L, V] rows of dtype logits_dtype (HYDRA_F32 or
 *           HYDRA_BF16), row stride ld >= V elements; row s*L + t holds the logits that
 *           predict ids[s*L + t] (already shifted by the caller).
 *   ids     : int32 [S*L] sampled token ids in [0, V).
 *   lengths : int32 [S] valid response tokens per sequence, 0..L; NULL means all L.
 *   seq_score : fp32 [S] sequence score added at t = len - 1; NULL means none.
 *   logp_actor, logp_ref, reward_tok : fp32 [S*L] outputs; rows t >= len are written 0
 *           and their logits are not read.
 *   lse_actor, lse_ref : optional fp32 [S*L] outputs (NULL to skip).
 * Requirements: S, L >= 0, 1 <= V < 2^31, ld >= V, S*L < 2^31.
 */
hydra_status hydra_token_logprobs_kl(const void* logits_actor, const void* logits_ref,
                                     int logits_dtype, int64_t S, int64_t L, int64_t V, int64_t ld,
                                     const int32_t* ids, const int32_t* lengths,
                                     const float* seq_score, float beta, float* logp_actor,
                                     float* logp_ref, float* reward_tok, float* lse_actor,
                                     float* lse_ref, void* stream);

/*
 * The dual LM head and the log-probabilities in one pass, without materialising logits:
 * equal to hydra_lora_linear(h_off, h_on, ..., W_lm, A, B, r, s, z_ref, z_actor, HYDRA_F32)
 * followed by hydra_token_logprobs_kl(z_actor, z_ref, ...), up to the fp32 summation order.
 * The tcgen05 GEMM's epilogue reduces each [row x 256-column] logit tile to a (max, sum exp)
 * pair and keeps the sampled token's logit; a second kernel merges the pairs into lse.
 * Arguments:
 *   h_off, h_on : bf16 [S*L, d] final hidden states of the reference (LoRA off) and actor
 *           (LoRA on) streams; h_on == h_off or NULL when they share the input.
 *   W : bf16 [V, d] LM head. A [r, d], B [V, r], r, s : LoRA of the actor head (r == 0: none).
 *   ids, lengths, seq_score, beta, logp_actor, logp_ref, reward_tok, lse_actor, lse_ref : as
 *           hydra_token_logprobs_kl with ids dense [S*L].
 *   workspace : hydra_lm_head_logprobs_workspace_size(S, L, V, r) bytes, 16-byte aligned
 *           (per-tile partials, sampled-token logits and u).
 * Errors: NULL required pointer -> HYDRA_ERR_NULL; d, V, r not multiples of 8 or a
 * misaligned pointer -> HYDRA_ERR_ALIGN; d < 8, V < 8, r > 256, S*L >= 2^31 ->
 * HYDRA_ERR_SHAPE; small workspace -> HYDRA_ERR_WORKSPACE. S*L == 0 is a no-op.
 */
size_t hydra_lm_head_logprobs_workspace_size(int64_t S, int64_t L, int64_t V, int64_t r);
hydra_status hydra_lm_head_logprobs(const void* h_off, const void* h_on, int64_t S, int64_t L,
                                    int64_t d, int64_t V, const void* W, const void* A,
                                    const void* B, int64_t r, float s, const int32_t* ids,
                                    const int32_t* lengths, const float* seq_score, float beta,
                                    float* logp_actor, float* logp_ref, float* reward_tok,
                                    float* lse_actor, float* lse_ref, void* workspace,
                                    size_t workspace_bytes, void* stream);

/*
 * Generalised advantage estimation over each sequence's valid tokens (§2: GAE uses
 * V(x, y) to build the advantage estimates and the critic regresses the returns;
 * Appendix B: gamma = 1.0, lambda = 0.95):
 *     delta_t = r_t + gamma V_{t+1} - V_t      (V_len = 0: terminal)
 *     A_t     = delta_t + gamma lambda A_{t+1} (A_len = 0)
 *     R_t     = A_t + V_t
 * rewards, values, advantages, returns : fp32 [S, L]; lengths : int32 [S] in 0..L or NULL
 * (all L). Positions t >= len are written 0. Requirements: S >= 0, 0 <= L <= 16384,
 * S*L < 2^40; outputs must not alias inputs.
 */
hydra_status ppo_gae(const float* rewards, const float* values, const int32_t* lengths, int64_t S,
                     int64_t L, float gamma, float lam, float* advantages, float* returns,
                     void* stream);

/*
 * Update side of PPO over a scored batch (§2 "Stage 3: PPO": probability ratio r(theta),
 * clipped surrogate L^CLIP, squared-error value loss on the returns; Algorithms 1 and 2
 * optimise this surrogate after scoring). Per valid token t < len_s:
 *     r_t = exp(logp_new_t - logp_old_t)
 *     A_t = advantages_t, or with whiten = 1: (advantages_t - mean) / sqrt(M2 / n + 1e-8),
 *           (n, mean, M2) the count, mean and sum of squared deviations of the valid
 *           advantages (population variance M2 / n)
 *     s_t = min(r_t A_t, clip(r_t, 1 - clip_eps, 1 + clip_eps) A_t)
 * Outputs (all n-normalised; n from the moments):
 *     grad_logp   fp32 [S, L]: d loss_clip / d logp_new = -r_t A_t / n where r_t A_t is the
 *                 smaller term (ties included), else 0; 0 at t >= len_s
 *     grad_values fp32 [S, L]: d loss_value / d values = 2 (values_t - returns_t) / n; 0 at
 *                 t >= len_s
 *     stats fp64 [7], device: [0] loss_clip = -(1/n) sum s_t, [1] loss_value = (1/n) sum
 *                 (values_t - returns_t)^2, [2] share of valid tokens with |r_t - 1| >
 *                 clip_eps, [3] approx KL (1/n) sum (logp_old_t - logp_new_t), [4] mean and
 *                 [5] population standard deviation of the raw advantages, [6] n.
 * The paper gives no clip range; clip_eps = 0.2 is the usual choice. A_t is a constant of
 * the loss (no gradient flows into the advantages).
 * Inputs logp_new, logp_old, advantages, returns, values: fp32 [S, L] row-major (row stride
 * L), device; lengths int32 [S] in 0..L, or NULL for all L (out of range: clamped, device
 * error 0x202). adv_moments: NULL, or device fp64 [3] = (n, mean, M2) to use instead of
 * this batch's own (e.g. merged over data-parallel replicas); n then also normalises the
 * losses and gradients, so replicas' losses add up to the global mean.
 * Reductions: compensated (Kahan) fp32 within a thread, fp32 trees across threads and
 * blocks, in a fixed order: results are bitwise reproducible for a given device and
 * accurate to a few fp32 ulps of the sums of magnitudes; the fp64 outputs carry those
 * values. exp overflows to inf for logp_new - logp_old
 * > 88.
 * workspace: device, 16-byte aligned, >= hydra_ppo_workspace_size() bytes, caller-owned;
 * no initial contents required; calls sharing a workspace must be stream-ordered.
 * Errors: NULL stats, or (S * L > 0) a NULL array -> HYDRA_ERR_NULL; S, L < 0 or S * L >= 2^31 ->
 * HYDRA_ERR_SHAPE; clip_eps outside [0, 1) or whiten not 0/1 -> HYDRA_ERR_RANGE; small or
 * misaligned workspace -> HYDRA_ERR_WORKSPACE. S * L == 0 writes stats of an empty batch
 * (all 0). Outputs must not alias inputs.
 */
size_t hydra_ppo_workspace_size(void);
hydra_status hydra_ppo_loss(const float* logp_new, const float* logp_old, const float* advantages,
                            const float* returns, const float* values, const int32_t* lengths,
                            int64_t S, int64_t L, float clip_eps, int whiten,
                            const double* adv_moments, float* grad_logp, float* grad_values,
                            double* stats, void* workspace, size_t workspace_bytes, void* stream);

/* (n, mean, M2) of the valid advantages of an [S, L] batch (the moments hydra_ppo_loss
 * whitens with), written to device fp64 [3] moments. Replicas merge their triples with the
 * pairwise update of Chan, Golub and LeVeque (1979) and pass the result to hydra_ppo_loss
 * as adv_moments. Arguments, workspace and errors as hydra_ppo_loss. */
hydra_status hydra_ppo_adv_moments(const float* advantages, const int32_t* lengths, int64_t S,
                                   int64_t L, double* moments, void* workspace,
                                   size_t workspace_bytes, void* stream);

/* Host-side merge of k moment triples (host fp64 [k][3] of (n, mean, M2), e.g. one per
 * data-parallel replica, gathered in rank order) into one host fp64 [3] triple, by the
 * pairwise update of Chan, Golub and LeVeque (1979) applied left to right:
 *     n = na + nb,  mean = mean_a + d nb / n,  M2 = M2a + M2b + d^2 na nb / n,
 * d = mean_b - mean_a. No device work. Errors: k < 0 -> HYDRA_ERR_SHAPE; NULL out (or NULL
 * moments with k > 0) -> HYDRA_ERR_NULL; a negative or NaN n or M2 -> HYDRA_ERR_RANGE. */
hydra_status hydra_ppo_merge_moments(const double* moments, int64_t k, double* out);

/* ===================================================================================
 * Llama decoder pieces and the full scoring pass (the paper runs Llama 7b, §4; the pass
 * follows the scoring steps of Algorithm 1, J-Hydra-PPO). The LoRA-off and LoRA-on streams
 * are stacked row-wise: rows [0, T) are the off stream, rows [T, 2T) the on stream, where
 * T = S * P for S sequences of P tokens. Residual stream fp32, matmul operands bf16.
 * =================================================================================== */

/* h[(c T + t), :] = table[ids[t], :] (bf16 -> fp32) for every copy c < copies.
 * table bf16 [V, d], ids int32 [T] in [0, V) (out of range: NaN row + device error),
 * h fp32 [copies * T, d]. d % 8 == 0. */
hydra_status hydra_embed(const void* table, int64_t V, int64_t d, const int32_t* ids, int64_t T,
                         int copies, float* h, void* stream);

/* RMSNorm (Zhang & Sennrich 2019): y[i] = bf16(x[j] / sqrt(mean(x[j]^2) + eps) * w) with
 * row gather j = (i / g_out) * g_in + off + i % g_out (g_out = g_in = rows, off = 0 for the
 * identity). x fp32 [*, d], w bf16 [d], y bf16 [rows, d]. d % 8 == 0. */
hydra_status hydra_rmsnorm(const float* x, const void* w, int64_t rows, int64_t d, float eps,
                           int64_t g_out, int64_t g_in, int64_t off, void* y, void* stream);

/* Rotary embedding (Su et al. 2021), rotate-half pairing, in place on the q block
 * (columns [0, d)) and k block ([d, 2d)) of each row of qkv (bf16 [R, ld]): dims (i, i + Dh/2)
 * of every head rotate by pos * theta^(-2i/Dh), pos = row % P. head_dim % 4 == 0, ld even. */
hydra_status hydra_rope(void* qkv, int64_t R, int64_t ld, int64_t d, int64_t head_dim, int64_t P,
                        float theta, void* stream);

/* Causal attention, out = softmax(q k^T / sqrt(Dh) + causal mask) v per head, for nseq
 * sequences of P rows each: q, k, v are column blocks [0, d), [d, 2d), [2d, 3d) of qkv
 * (bf16, row stride ld), out bf16 with row stride ld_out. head_dim must be 128; ld and
 * ld_out multiples of 8, qkv and out 16-byte aligned (else HYDRA_ERR_ALIGN). Runs on the
 * tcgen05 tensor cores with the probabilities rounded to bf16 before the P V product. */
hydra_status hydra_causal_attention(const void* qkv, int64_t nseq, int64_t P, int64_t ld,
                                    int64_t n_heads, int64_t head_dim, void* out, int64_t ld_out,
                                    void* stream);

/* SwiGLU (Shazeer 2020): m = bf16(silu(g) * u), gu bf16 [R, 2F] = [gate | up], m [R, F]. */
hydra_status hydra_swiglu(const void* gu, int64_t R, int64_t F, void* m, void* stream);

/* h += float(y) over n elements (h fp32, y bf16, n % 8 == 0). */
hydra_status hydra_residual_add(float* h, const void* y, int64_t n, void* stream);

/* Scalar head (reward model / value head): out[i] = sum_k x[j, k] w[k] with the row gather
 * of hydra_rmsnorm. x bf16, w bf16 [d], out fp32 [n]. */
hydra_status hydra_head_dot(const void* x, int64_t d, const void* w, int64_t n, int64_t g_out,
                            int64_t g_in, int64_t off, float* out, void* stream);

typedef struct hydra_llama_config {
  int64_t n_layers, d_model, n_heads, head_dim, ffn, vocab;
  int64_t prompt_len;   /* P0: prompt tokens per sequence */
  int64_t response_len; /* L: response slots per sequence (each sequence is P0 + L tokens) */
  int64_t lora_rank;    /* r of every adapted linear (q, v, gate, up, down) */
  float lora_scale, rms_eps, rope_theta;
  float beta, gamma, lam; /* KL coefficient, GAE discount and lambda */
} hydra_llama_config;

/* One decoder layer, fused layouts (device pointers, bf16):
 *   w_qkv [3d, d] = [Wq; Wk; Wv]        a_qv [2r, d] = [Aq; Av]
 *   b_qkv [3d, 2r] = [[Bq, 0]; [0, 0]; [0, Bv]]   (LoRA on q and v only)
 *   w_o [d, d] (no LoRA)
 *   w_gu [2F, d]: gate and up rows interleaved in blocks of 128 (block 2j = gate rows
 *        128j..128j+127, block 2j+1 = up rows of the same features); F % 128 == 0
 *   a_gu [2r, d] = [A_gate; A_up]
 *   b_gu [2F, 2r]: rows interleaved like w_gu; gate rows [B_gate_row, 0], up rows
 *        [0, B_up_row]
 *   w_down [d, F], a_down [r, F], b_down [d, r]
 *   norm_attn, norm_ffn [d] */
typedef struct hydra_llama_layer {
  const void* w_qkv;
  const void* a_qv;
  const void* b_qkv;
  const void* w_o;
  const void* w_gu;
  const void* a_gu;
  const void* b_gu;
  const void* w_down;
  const void* a_down;
  const void* b_down;
  const void* norm_attn;
  const void* norm_ffn;
} hydra_llama_layer;

typedef struct hydra_llama_weights {
  const void* embed;               /* bf16 [V, d] */
  const hydra_llama_layer* layers; /* HOST array of n_layers entries */
  const void* final_norm;          /* bf16 [d] */
  const void* lm_head;             /* bf16 [V, d] */
  const void* w_rm;                /* bf16 [d]: reward-model head; also the value head */
} hydra_llama_weights;

/* One LoRA set of a decoder layer in the fused layouts of hydra_llama_layer (the critic's
 * set of Hydra-PPO): a_qv [2r, d] / b_qkv [3d, 2r] (q and v adapted, k not), a_gu [2r, d] /
 * b_gu [2F, 2r] (interleaved gate/up rows), a_down [r, F] / b_down [d, r]. */
typedef struct hydra_llama_lora {
  const void* a_qv;
  const void* b_qkv;
  const void* a_gu;
  const void* b_gu;
  const void* a_down;
  const void* b_down;
} hydra_llama_lora;

/* Workspace bytes of hydra_generate_llama for S sequences (0 for an unsupported
 * configuration or S outside 1..64). */
size_t hydra_generate_llama_workspace_size(const hydra_llama_config* cfg, int64_t S);

/*
 * Generation with the actor (Algorithms 1 and 2: the actor samples each sequence for T steps;
 * J-Hydra-PPO keeps the critic head's values while sampling), KV-cached, with
 * the LoRA-off stream decoded beside the actor so that each drawn token also gets its
 * reference log-probability (one read of W serves both streams' rows).
 * For each of S sequences of P0 = cfg->prompt_len prompt tokens and steps t < n_steps:
 *   z_on, z_off = LM head of the final normed hidden state at position P0 + t - 1 of the
 *                 LoRA-on and LoRA-off streams (fp32 logits)
 *   tokens[s, t]     = argmax_k (z_on[k] + gumbel[t, s, k])   (greedy argmax if gumbel is
 *                      NULL; ties to the lowest k). With standard Gumbel noise this is a
 *                      draw from softmax(z_on) (Gumbel-max); the noise is the caller's.
 *   logp_actor[s, t] = log_softmax(z_on)[token],  logp_ref[s, t] = log_softmax(z_off)[token]
 *   values[s, t]     = w_rm . h_on at position P0 + t - 1 (J-Hydra: r_phi = LO(V))
 *   score[s]         = w_rm . h_off at position P0 + n_steps - 1 (the reward model on the
 *                      state after the last drawn token; one more decode pass), if score
 *                      is not NULL.
 * These equal hydra_score_llama's logp_actor, logp_ref, values and score on the finished
 * sequence (prompt + tokens). Weights as hydra_score_llama (fused layouts).
 * prompt_ids int32 [S, P0]; gumbel fp32 [n_steps, S, V] or NULL; outputs int32 / fp32
 * [S, n_steps] and fp32 [S]; all device. Requirements: as hydra_score_llama, plus
 * 1 <= S <= 64, 1 <= n_steps <= cfg->response_len (the cache holds P0 + response_len
 * positions; its scores fit shared memory for P0 + response_len up to about 50,000).
 * workspace: device, 16-byte aligned, >= hydra_generate_llama_workspace_size(cfg, S).
 * Errors: NULL pointer -> HYDRA_ERR_NULL; configuration or sizes outside the above ->
 * HYDRA_ERR_SHAPE; misaligned weight or workspace -> HYDRA_ERR_ALIGN; small workspace ->
 * HYDRA_ERR_WORKSPACE; token id out of range -> device error 0x201.
 */
hydra_status hydra_generate_llama(const hydra_llama_config* cfg, const hydra_llama_weights* w,
                                  const int32_t* prompt_ids, int64_t S, int64_t n_steps,
                                  const float* gumbel, void* workspace, size_t workspace_bytes,
                                  int32_t* tokens, float* logp_actor, float* logp_ref,
                                  float* values, float* score, void* stream);

/* Workspace bytes of hydra_score_llama for S sequences. */
size_t hydra_score_llama_workspace_size(const hydra_llama_config* cfg, int64_t S);

/*
 * The full J-Hydra scoring pass (Algorithm 1: the LoRA-off model gives the reference
 * log-probabilities and the reward; §3 Dynamic LoRA; J-Hydra uses one LoRA set for actor
 * and critic) over S sequences of P0 prompt + L response tokens:
 *   both streams through n_layers Llama blocks (q/v/gate/up/down carry LoRA, k/o/LM head
 *   do not) -> final RMSNorm -> LM head on the rows predicting response tokens, reduced
 *   in its epilogue to log-softmax partials (as hydra_lm_head_logprobs; no logits are
 *   stored) -> logp_actor (LoRA on), logp_ref (LoRA off) -> score_s = w_rm . h_off[P0 + len_s - 1],
 *   values_t = w_rm . h_on[P0 + t - 1] -> reward_t = -beta (la - lr) + [t = len-1] score
 *   -> GAE advantages and returns.
 * ids int32 [S, P0 + L]; lengths int32 [S] valid response tokens (0..L) or NULL (all L).
 * Outputs fp32 [S, L] (0 at t >= len): logp_actor, logp_ref, reward, values, advantages,
 * returns; score fp32 [S]. Requirements: head_dim == 128, d == n_heads * 128,
 * ffn % 128 == 0, vocab % 8 == 0, r % 8 == 0, 8 <= r <= 128, P0 >= 1, L >= 1.
 * Work skipped because nothing reads it: layer 0's q/k/v products are formed once for both
 * streams (their inputs are equal there), and the last layer's o projection and feed-forward
 * block run only on positions P0 - 1 .. P0 + L - 1 of each sequence, the rows the heads read.
 */
hydra_status hydra_score_llama(const hydra_llama_config* cfg, const hydra_llama_weights* w,
                               const int32_t* ids, const int32_t* lengths, int64_t S,
                               void* workspace, size_t workspace_bytes, float* logp_actor,
                               float* logp_ref, float* reward, float* values, float* advantages,
                               float* returns, float* score, void* stream);

/*
 * The Hydra-PPO scoring pass (Algorithm 2; §3 Stage 2: two LoRA sets on one base model):
 * as hydra_score_llama with three stacked streams through every layer (layer 0 included; the
 * last layer on the rows the heads read), each W read once for
 * all three (hydra_lora_linear_tri): LoRA off (reference log-probabilities, reward score),
 * the actor's LoRA set w->layers (logp_actor) and the critic's LoRA set critic[l] (a HOST
 * array of n_layers entries, same rank r), whose final hidden states give the values through
 * the reward head (r_phi <- LO(V)): values_t = w_rm . h_critic[P0 + t - 1]. With critic equal
 * to the actor's LoRA pointers the outputs equal hydra_score_llama's (J-Hydra-PPO).
 * Workspace: hydra_score_llama_hydra_workspace_size(cfg, S); other arguments and errors as
 * hydra_score_llama; NULL critic -> HYDRA_ERR_NULL.
 */
size_t hydra_score_llama_hydra_workspace_size(const hydra_llama_config* cfg, int64_t S);
hydra_status hydra_score_llama_hydra(const hydra_llama_config* cfg, const hydra_llama_weights* w,
                                     const hydra_llama_lora* critic, const int32_t* ids,
                                     const int32_t* lengths, int64_t S, void* workspace,
                                     size_t workspace_bytes, float* logp_actor, float* logp_ref,
                                     float* reward, float* values, float* advantages,
                                     float* returns, float* score, void* stream);

/* Kernel classes of the optional launch timing of hydra_score_llama. */
enum {
  HYDRA_PROF_GEMM_QKV = 0,    /* tcgen05 dual-output linears: fused q/k/v */
  HYDRA_PROF_GEMM_O = 1,      /* o projection (+ residual add epilogue) */
  HYDRA_PROF_GEMM_GU = 2,     /* fused gate/up (+ SwiGLU epilogue) */
  HYDRA_PROF_GEMM_DOWN = 3,   /* down projection (+ residual add epilogue) */
  HYDRA_PROF_GEMM_LMHEAD = 4, /* LM head with the log-softmax partials in its epilogue */
  HYDRA_PROF_LORA_DOWN = 5,   /* u = s x A^T */
  HYDRA_PROF_ATTENTION = 6,   /* causal attention */
  HYDRA_PROF_ELEMENTWISE = 7, /* embedding, RMSNorm, RoPE */
  HYDRA_PROF_LOGPROBS = 8,    /* log-softmax + gather + KL reward */
  HYDRA_PROF_GAE = 9,         /* GAE scan */
  HYDRA_PROF_HEADS = 10,      /* reward-model score and value head */
  HYDRA_PROF_CLASSES = 11
};

/*
 * Launch timing of hydra_score_llama. While enabled, every kernel launch of the pass is
 * bracketed by CUDA events recorded on the call's stream (host-side overhead only; the
 * events come from a library pool created on first use). hydra_profile_collect waits for
 * the recorded events, writes the summed milliseconds and launch counts per class into
 * ms[HYDRA_PROF_CLASSES] and launches[HYDRA_PROF_CLASSES] (host arrays), and with reset
 * != 0 starts a new collection. This is measurement support, not part of the paper.
 */
hydra_status hydra_profile_enable(int on);
hydra_status hydra_profile_collect(float* ms, int64_t* launches, int reset);

#ifdef __cplusplus
}
#endif

#endif /* HYDRA_H_ */
