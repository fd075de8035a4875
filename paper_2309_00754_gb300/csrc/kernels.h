// Internal launch interface between the C-ABI layer (api.cu) and the kernel files.
// Every launcher validates nothing: api.cu has checked pointers, sizes and alignment.
// Launchers return 0 on success, a negative code when a launch or a tensor-map encode
// failed.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace hydra {

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
};

int launch_dual_lora_gemm_tc(const GemmArgs& a, cudaStream_t stream);
int launch_dual_lora_gemv(const GemmArgs& a, cudaStream_t stream);
int launch_lora_down(const void* x, int64_t M, int64_t K, const void* A, int64_t r, float s,
                     void* u, cudaStream_t stream);
int launch_token_logprobs_kl(const void* za, const void* zr, int bf16_logits, int64_t S, int64_t L,
                             int64_t V, int64_t ld, const int32_t* ids, const int32_t* lengths,
                             const float* score, float beta, float* la, float* lr, float* rew,
                             float* lse_a, float* lse_r, int* err, cudaStream_t stream);
int launch_gae(const float* r, const float* v, const int32_t* lengths, int64_t S, int64_t L,
               float gamma, float lam, float* adv, float* ret, int* err, cudaStream_t stream);

// Largest sequence length the shared-memory GAE scan accepts.
constexpr int64_t kGaeMaxL = 16384;
// Largest number of token rows (both streams together) the GEMV path takes.
constexpr int64_t kGemvMaxRows = 16;

}  // namespace hydra
