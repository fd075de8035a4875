// Internal launch interface between the C-ABI layer (api.cu) and the kernel files.
// Every launcher validates nothing: api.cu has checked pointers, sizes and alignment.
// Launchers return 0 on success, a negative code when a launch or a tensor-map encode
// failed.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <utility>

namespace hydra {

// Launch with programmatic stream serialisation: the kernel may begin while the preceding
// kernel of the stream finishes, and must call pdl_wait() (common.cuh) before reading
// anything that work may write or writing anything.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t stream, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

struct GemmArgs {
  const void* x_off;  // bf16 [M, K]
  const void* x_on;   // bf16 [M, K] (ignored when shared_x)
  int64_t M, K, N;
  const void* W;      // bf16 [N, K]
  const void* u;      // bf16 [M, r] = s * x_on A^T (NULL when r == 0)
  const void* B;      // bf16 [N, r]
  int64_t r;
  bool shared_x;
  void* y_off;        // [M, N] bf16 or fp32, may be NULL
  void* y_on;         // [M, N] bf16 or fp32, may be NULL
  int out_f32;
  int* err;
  // third stream (Hydra-PPO critic): input, LoRA operands (same r as the on stream) and
  // output; NULL x_crit means two streams
  const void* x_crit = nullptr;
  const void* u_crit = nullptr;
  const void* B_crit = nullptr;
  void* y_crit = nullptr;
  int epi = 0;        // tcgen05 epilogue: 0 store, 1 SwiGLU, 2 residual add (fp32), 3 rotary,
                      // 4 log-softmax partials
  bool single_cta = false;  // tcgen05: never use the CTA-pair (cta_group::2) kernel
  // epi 3 (rotary): columns [0, rope_cols) rotate in heads of 128 at position row % rope_P,
  // by the (cos, sin) pairs of rope_table [rope_P][64] (launch_rope_table)
  int64_t rope_P = 1;
  int64_t rope_cols = 0;
  const void* rope_table = nullptr;
  // epi 4 (log-softmax partials): y_off / y_on are float2 [M][ceil(N / 256)] partial
  // (max, sum exp) arrays, lsm_target float [2][M] the sampled-token logits, and the token of
  // row m is lsm_ids[(m / lsm_L) * lsm_ids_ld + lsm_ids_off + m % lsm_L]
  float* lsm_target = nullptr;
  const int32_t* lsm_ids = nullptr;
  int64_t lsm_L = 1, lsm_ids_ld = 1, lsm_ids_off = 0;
};

// Device address of the library's error word on the current device (NULL on failure).
int* device_error_word();

int launch_dual_lora_gemm_tc(const GemmArgs& a, cudaStream_t stream);
// TMA map over a row-major [rows, cols] bf16 (or fp32) matrix with row stride ld elements:
// 128-byte swizzle, boxes of [box_rows x 128 bytes], zero fill out of bounds
bool make_tma_map(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int64_t ld,
                  int box_rows, bool f32);
// TMA map over bf16 planes of [rows, cols] (row stride ld, plane stride plane_stride elements):
// 128-byte swizzle, boxes of [box_rows x 64] in one plane; out-of-range elements are not
// written by a store
bool make_tma_map_3d(CUtensorMap* map, const void* base, int64_t cols, int64_t rows,
                     int64_t planes, int64_t ld, int64_t plane_stride, int box_rows);
int launch_dual_lora_gemv(const GemmArgs& a, cudaStream_t stream);

// Skinny linear (gemm_skinny.cu): y = x W^T for all M <= 128 rows of x, plus u B^T on rows
// [u_row0, u_row0 + u_rows) (u [u_rows, r]). K is split over a cluster of ks CTAs; bn / ks
// of 0 pick them by the kernel's cost model. Needs K % 8 == 0, N % 16 == 0, r % 8 == 0.
struct SkinnyArgs {
  const void* x;  // bf16 [M, K]
  int64_t M, K, N;
  const void* W;  // bf16 [N, K]
  const void* u;  // bf16 [u_rows, r] (NULL when r == 0)
  int64_t u_row0, u_rows;
  const void* B;  // bf16 [N, r]
  int64_t r;
  void* y;        // [M, N], bf16 or fp32 (out_f32)
  int out_f32;
  int bn, ks;     // 0 = chosen by the cost model
  int* err;
};
bool skinny_gemm_supported(int64_t M, int64_t K, int64_t N, int64_t r);
int launch_skinny_gemm_tc(const SkinnyArgs& a, cudaStream_t stream);
int launch_lora_down(const void* x, int64_t M, int64_t K, const void* A, int64_t r, float s,
                     void* u, cudaStream_t stream);
// ids of sequence s start at ids + s * ids_ld (ids_ld = L for a dense [S, L] array)
// merge the per-tile (max, sum exp) partials [rows][n_tiles] (float2) of the reference and
// actor heads and their sampled-token logits [rows] into logp / reward (as
// launch_token_logprobs_kl); ids of sequence s start at ids + s * ids_ld
int launch_lse_combine(const void* part_ref, const void* part_act, int64_t n_tiles,
                       const float* tgt_ref, const float* tgt_act, int64_t S, int64_t L, int64_t V,
                       const int32_t* ids, int64_t ids_ld, const int32_t* lengths,
                       const float* score, float beta, float* la, float* lr, float* rew,
                       float* lse_a, float* lse_r, int* err, cudaStream_t stream);
int launch_token_logprobs_kl(const void* za, const void* zr, int bf16_logits, int64_t S, int64_t L,
                             int64_t V, int64_t ld, const int32_t* ids, int64_t ids_ld,
                             const int32_t* lengths,
                             const float* score, float beta, float* la, float* lr, float* rew,
                             float* lse_a, float* lse_r, int* err, cudaStream_t stream);
int launch_gae(const float* r, const float* v, const int32_t* lengths, int64_t S, int64_t L,
               float gamma, float lam, float* adv, float* ret, int* err, cudaStream_t stream);

// PPO update-side losses (ppo_loss.cu). ext_moments (device [n, mean, M2]) or NULL.
size_t ppo_loss_workspace_bytes();
int launch_ppo_adv_moments(const float* adv, const int32_t* lengths, int64_t S, int64_t L,
                           double* out, void* ws, int* err, cudaStream_t st);
int launch_ppo_loss(const float* logp_new, const float* logp_old, const float* adv,
                    const float* ret, const float* val, const int32_t* lengths, int64_t S,
                    int64_t L, float eps, bool whiten, const double* ext_moments,
                    float* grad_logp, float* grad_val, double* stats, void* ws, int* err,
                    cudaStream_t st);
// Blocks of the two PPO passes (one fp64 partial per block lives in the workspace).
constexpr int kPpoMaxMomentBlocks = 1024;
constexpr int kPpoMaxLossBlocks = 1024;

// The full pass's stacked linear over ns row-stacked streams (score_llama.cu): rows [0, T)
// of x are the LoRA-off stream, [T, 2T) the LoRA-on stream (LoRA set A, B; u receives its
// down-projection) and, for ns == 3, [2T, 3T) a third stream with the set A2, B2 (u2). epi:
// HYDRA_EPI_* or kStackEpiRope with rope's arguments; y as the tcgen05 GEMM's epilogue
// writes it. prof_class: the HYDRA_PROF_* class its launches are timed under.
constexpr int kStackEpiRope = 3;
struct StackRope {
  int64_t P, cols;
  const void* table;  // (cos, sin) [P][head_dim / 2]
};
int stacked_linear(int prof_class, const void* x, int64_t T, int64_t K, int64_t N, const void* W,
                   const void* A, const void* B, int64_t r, float s, void* u, void* y, bool f32,
                   int* err, cudaStream_t st, int epi = 0, const StackRope* rope = nullptr,
                   int ns = 2, const void* A2 = nullptr, const void* B2 = nullptr,
                   void* u2 = nullptr);

// Generation loop kernels (decode.cu). Cache per layer: K then V, each [R][H][Pmax][128]
// bf16; step: device counter of the current draw (the new token sits at P0 + step - 1).
int launch_kv_store_prefill(const void* qkv, int64_t R, int64_t P0, int64_t ld, int64_t d,
                            int64_t H, int64_t Pmax, void* ck, void* cv, cudaStream_t st);
size_t decode_attention_smem(int64_t Pmax);
// rotary of the new token's q and k (table [Pmax][64] (cos, sin)), its k and v appended to
// the cache at P0 + step - 1, then attention of q over the cached positions
int launch_decode_attention(void* qkv, int64_t R, int64_t ld, int64_t d, int64_t H,
                            const void* table, void* ck, void* cv, int64_t P0, const int* step,
                            int64_t Pmax, void* out, int64_t ld_out, cudaStream_t st);
int launch_sample_tokens(const float* logits, int64_t S, int64_t V, const float* gumbel,
                         const void* fin, int64_t d, const void* w_rm, const int* step,
                         int64_t n_steps, int32_t* tokens, float* logp_a, float* logp_r,
                         float* values, int32_t* cur_ids, cudaStream_t st);
// Thread-block-cluster row kernels of the decode step (8 CTAs per row): h += y (y may be
// NULL), a = bf16(rmsnorm(h) w) and, for rows i >= S, u[i - S] = bf16(s a A^T) (A [r2, d] or
// NULL); and m = SwiGLU(gu) (gate/up interleaved by 128) with u[i - S] = bf16(s m A^T).
int launch_row_norm_lora(float* h, const void* y, const void* w, int64_t R, int64_t d, float eps,
                         void* a, int64_t S, const void* A, int64_t r2, float s, void* u,
                         cudaStream_t st);
int launch_swiglu_lora(const void* gu, int64_t R, int64_t F, void* m, int64_t S, const void* A,
                       int64_t r, float s, void* u, cudaStream_t st);

// Row gather used by the per-row Llama kernels: output row i reads input row
// (i / g_out) * g_in + off + i % g_out (g_out = g_in, off = 0 is the identity).
struct RowMap {
  long long g_out, g_in, off;
};

// h [copies T, d] fp32 = the embedding rows of ids; with `step` (decode), a dependent launch
// that also advances the device-side step counter by one
int launch_embed(const void* table, int64_t V, int64_t d, const int32_t* ids, int64_t T,
                 int copies, float* h, int* err, cudaStream_t st, int* step = nullptr);
int launch_rmsnorm(const float* x, const void* w, int64_t rows, int64_t d, float eps,
                   const RowMap& map, void* y, cudaStream_t st);
// (cos, sin) float2 table [P][Dh / 2] of the rotary angles pos * theta^(-2i/Dh)
int launch_rope_table(int64_t P, int64_t Dh, float theta, void* table, cudaStream_t st);
int launch_rope(void* qkv, int64_t R, int64_t ld, int64_t d, int64_t Dh, int64_t P, float theta,
                cudaStream_t st);
int launch_swiglu(const void* gu, int64_t R, int64_t F, void* m, cudaStream_t st);
int launch_residual_add(float* h, const void* y, int64_t n, cudaStream_t st);
int launch_head_dot(const void* x, int64_t d, const void* w, const RowMap& map, int64_t n,
                    const int32_t* lengths, int64_t L, float* out, cudaStream_t st);
int launch_seq_score(const float* h, const void* norm, const void* w, int64_t d, float eps,
                     const int32_t* lengths, int64_t S, int64_t L, int64_t P, int64_t p0,
                     float* score, cudaStream_t st);
int launch_causal_attention(const void* qkv, int64_t nseq, int64_t P, int64_t ld, int64_t n_heads,
                            int64_t head_dim, void* out, int64_t ld_out, cudaStream_t st);
// dst row i = src row map(i) for i < rows, rows of row_bytes bytes (a multiple of 16)
int launch_gather_rows(const void* src, int64_t rows, int64_t row_bytes, const RowMap& map,
                       void* dst, cudaStream_t st);

// Largest sequence length the shared-memory GAE scan accepts.
constexpr int64_t kGaeMaxL = 16384;
// Largest number of token rows (both streams together) the GEMV path takes.
constexpr int64_t kGemvMaxRows = 16;

}  // namespace hydra
