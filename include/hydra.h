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
 *   2 GEMV (at most 16 token rows over both streams).
 * Same layout, alignment and error rules as hydra_lora_linear; no workspace.
 */
hydra_status hydra_dual_linear(const void* x_off, const void* x_on, int64_t M, int64_t K,
                               int64_t N, const void* W, const void* u, const void* B, int64_t r,
                               void* y_off, void* y_on, int out_dtype, int algo, void* stream);

/*
 * hydra_lora_linear with the kernel family chosen by the caller:
 *   algo 0 = automatic (as hydra_lora_linear), 1 = tcgen05 tile kernel (any M),
 *   2 = GEMV kernel (requires at most 16 token rows over both streams).
 * Same arguments, results and errors otherwise; algo outside 0..2 is HYDRA_ERR_RANGE.
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

#ifdef __cplusplus
}
#endif

#endif /* HYDRA_H_ */
