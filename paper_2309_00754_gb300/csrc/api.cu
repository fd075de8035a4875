// C-ABI entry points of libhydra (declared in include/hydra.h): argument validation on
// the host, then kernel launches on the caller's stream.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "../../include/hydra.h"
#include "common.cuh"
#include "kernels.h"

namespace {

// The library's device error word (one per device that loaded the library).
__device__ int g_hydra_err = 0;

constexpr int kMaxDevices = 64;
int* g_err_ptr[kMaxDevices] = {nullptr};
std::mutex g_err_ptr_mutex;  // guards the first fill of g_err_ptr from concurrent host threads

}  // namespace

namespace hydra {

// Device address of the library's error word on the current device (resolved once).
int* device_error_word() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_err_ptr_mutex);
  if (g_err_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_hydra_err) != cudaSuccess) return nullptr;
    g_err_ptr[dev] = static_cast<int*>(p);
  }
  return g_err_ptr[dev];
}

}  // namespace hydra

namespace {

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

inline size_t round_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// Rotary epilogue arguments (hydra_dual_linear_rope).
struct RopeArgs {
  int64_t P, cols, head_dim;
  const float* table;
};
constexpr int kEpiRope = 3;  // internal epilogue code of the rotary mode

// u_given: `workspace` already holds u = s x_on A^T (hydra_dual_linear); A is unused.
// epi: tcgen05 epilogue (store / SwiGLU / residual add / rotary); non-store epilogues need
// algo 1 or 3; rope carries the rotary arguments of epi == kEpiRope.
hydra_status lora_linear_impl(const void* x_off, const void* x_on, int64_t M, int64_t K,
                              int64_t N, const void* W, const void* A, const void* B, int64_t r,
                              float s, void* y_off, void* y_on, int out_dtype, void* workspace,
                              size_t workspace_bytes, int algo, void* stream,
                              bool u_given = false, int epi = HYDRA_EPI_STORE,
                              const RopeArgs* rope = nullptr) {
  if (x_off == nullptr || W == nullptr) return HYDRA_ERR_NULL;
  if (y_off == nullptr && y_on == nullptr) return HYDRA_ERR_NULL;
  if (algo < 0 || algo > 3) return HYDRA_ERR_RANGE;
  if (epi < HYDRA_EPI_STORE || epi > (rope != nullptr ? kEpiRope : HYDRA_EPI_RESIDUAL))
    return HYDRA_ERR_RANGE;
  if (epi == kEpiRope) {
    if (rope->table == nullptr) return HYDRA_ERR_NULL;
    if (!aligned16(rope->table)) return HYDRA_ERR_ALIGN;
    if (out_dtype != HYDRA_BF16 || rope->head_dim != 128) return HYDRA_ERR_RANGE;
    if (rope->P < 1 || rope->cols < 0 || rope->cols > N || rope->cols % 128 != 0) return HYDRA_ERR_SHAPE;
  }
  if (epi != HYDRA_EPI_STORE && algo != 1 && algo != 3) return HYDRA_ERR_RANGE;
  if (epi == HYDRA_EPI_SWIGLU && N % 256 != 0) return HYDRA_ERR_SHAPE;
  if (out_dtype != HYDRA_BF16 && out_dtype != HYDRA_F32) return HYDRA_ERR_RANGE;
  if (M < 0 || K < 8 || N < 8 || M >= (1LL << 31) || K >= (1LL << 31) || N >= (1LL << 31))
    return HYDRA_ERR_SHAPE;
  if (K % 8 != 0 || N % 8 != 0) return HYDRA_ERR_ALIGN;
  if (r < 0 || r > 256) return HYDRA_ERR_SHAPE;
  if (r > 0 && r % 8 != 0) return HYDRA_ERR_ALIGN;
  const bool shared_x = (x_on == nullptr || x_on == x_off);
  if (!aligned16(x_off) || (!shared_x && !aligned16(x_on)) || !aligned16(W) ||
      !aligned16(y_off) || !aligned16(y_on))
    return HYDRA_ERR_ALIGN;
  const bool lora = r > 0 && y_on != nullptr;
  if (lora) {
    if ((!u_given && A == nullptr) || B == nullptr) return HYDRA_ERR_NULL;
    if ((!u_given && !aligned16(A)) || !aligned16(B)) return HYDRA_ERR_ALIGN;
    if (workspace == nullptr) return u_given ? HYDRA_ERR_NULL : HYDRA_ERR_WORKSPACE;
    if (!aligned16(workspace)) return HYDRA_ERR_ALIGN;
    if (workspace_bytes < hydra_lora_linear_workspace_size(M, r)) return HYDRA_ERR_WORKSPACE;
  }
  const int64_t rows = shared_x ? M : 2 * M;
  if (algo == 2 && rows > hydra::kGemvMaxRows) return HYDRA_ERR_SHAPE;
  if (M == 0) return HYDRA_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int* err = hydra::device_error_word();
  if (err == nullptr) return HYDRA_ERR_CUDA;

  const void* xo = shared_x ? x_off : x_on;
  if (lora && !u_given) {
    if (hydra::launch_lora_down(xo, M, K, A, r, s, workspace, st) != 0) return HYDRA_ERR_CUDA;
  }
  hydra::GemmArgs g;
  g.x_off = x_off;
  g.x_on = xo;
  g.M = M;
  g.K = K;
  g.N = N;
  g.W = W;
  g.u = lora ? workspace : nullptr;
  g.B = lora ? B : nullptr;
  g.r = lora ? r : 0;
  g.shared_x = shared_x;
  g.y_off = y_off;
  g.y_on = y_on;
  g.out_f32 = out_dtype == HYDRA_F32 ? 1 : 0;
  g.err = err;
  g.epi = epi;
  g.single_cta = algo == 3;
  if (epi == kEpiRope) {
    g.rope_P = rope->P;
    g.rope_cols = rope->cols;
    g.rope_table = rope->table;
  }
  const bool use_gemv = (algo == 2) || (algo == 0 && rows <= hydra::kGemvMaxRows);
  const int rc = use_gemv ? hydra::launch_dual_lora_gemv(g, st) : hydra::launch_dual_lora_gemm_tc(g, st);
  return rc == 0 ? HYDRA_OK : HYDRA_ERR_CUDA;
}

// One warp waits on an mbarrier that nothing ever arrives on, through the bounded wait that
// every kernel of the library uses: the wait expires after kWaitBudgetCycles, records
// kDevTimeoutSelftest in the device error word and the kernel returns.
__global__ void bounded_wait_selftest_kernel(int* err) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    hydra::mbar_init(hydra::smem_u32(&bar), 1);
    abort_flag = 0;
    hydra::fence_mbar_init();
  }
  __syncthreads();
  hydra::warp_wait_bounded(hydra::smem_u32(&bar), 0, reinterpret_cast<volatile int*>(&abort_flag),
                           err, hydra::kDevTimeoutSelftest);
}

}  // namespace

extern "C" {

const char* hydra_status_string(int status) {
  switch (status) {
    case HYDRA_OK: return "HYDRA_OK";
    case HYDRA_ERR_NULL: return "HYDRA_ERR_NULL: a required pointer is NULL";
    case HYDRA_ERR_SHAPE: return "HYDRA_ERR_SHAPE: size out of the supported range";
    case HYDRA_ERR_ALIGN: return "HYDRA_ERR_ALIGN: pointer or row length not 16-byte aligned";
    case HYDRA_ERR_RANGE: return "HYDRA_ERR_RANGE: scalar or enum argument out of range";
    case HYDRA_ERR_CUDA: return "HYDRA_ERR_CUDA: CUDA runtime or driver call failed";
    case HYDRA_ERR_TIMEOUT: return "HYDRA_ERR_TIMEOUT: bounded device wait expired";
    case HYDRA_ERR_WORKSPACE: return "HYDRA_ERR_WORKSPACE: workspace missing or too small";
    case HYDRA_ERR_DEVICE: return "HYDRA_ERR_DEVICE: kernel found a bad token id or length";
    default: return "unknown hydra status";
  }
}

int hydra_abi_version(void) { return 1; }

hydra_status hydra_selftest_wait_timeout(void* stream) {
  int* err = hydra::device_error_word();
  if (err == nullptr) return HYDRA_ERR_CUDA;
  bounded_wait_selftest_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(err);
  return cudaPeekAtLastError() == cudaSuccess ? HYDRA_OK : HYDRA_ERR_CUDA;
}

hydra_status hydra_device_error(int32_t* code_out, int clear) {
  if (code_out == nullptr) return HYDRA_ERR_NULL;
  int v = 0;
  if (cudaDeviceSynchronize() != cudaSuccess) return HYDRA_ERR_CUDA;
  if (cudaMemcpyFromSymbol(&v, g_hydra_err, sizeof(int)) != cudaSuccess) return HYDRA_ERR_CUDA;
  if (clear) {
    const int zero = 0;
    if (cudaMemcpyToSymbol(g_hydra_err, &zero, sizeof(int)) != cudaSuccess) return HYDRA_ERR_CUDA;
  }
  *code_out = v;
  return HYDRA_OK;
}

size_t hydra_lora_linear_workspace_size(int64_t M, int64_t r) {
  if (M <= 0 || r <= 0) return 0;
  return round_up(static_cast<size_t>(M) * static_cast<size_t>(r) * 2, 256);
}

hydra_status hydra_lora_down(const void* x_on, int64_t M, int64_t K, const void* A, int64_t r,
                             float s, void* u, void* stream) {
  if (x_on == nullptr || A == nullptr || u == nullptr) return HYDRA_ERR_NULL;
  if (M < 0 || K < 8 || r < 1 || r > 256 || M >= (1LL << 31) || K >= (1LL << 31))
    return HYDRA_ERR_SHAPE;
  if (K % 8 != 0 || r % 8 != 0) return HYDRA_ERR_ALIGN;
  if (!aligned16(x_on) || !aligned16(A) || !aligned16(u)) return HYDRA_ERR_ALIGN;
  if (M == 0) return HYDRA_OK;
  return hydra::launch_lora_down(x_on, M, K, A, r, s, u, static_cast<cudaStream_t>(stream)) == 0
             ? HYDRA_OK
             : HYDRA_ERR_CUDA;
}

hydra_status hydra_lora_linear(const void* x_off, const void* x_on, int64_t M, int64_t K,
                               int64_t N, const void* W, const void* A, const void* B, int64_t r,
                               float s, void* y_off, void* y_on, int out_dtype, void* workspace,
                               size_t workspace_bytes, void* stream) {
  return lora_linear_impl(x_off, x_on, M, K, N, W, A, B, r, s, y_off, y_on, out_dtype, workspace,
                          workspace_bytes, 0, stream);
}

hydra_status hydra_lora_linear_algo(const void* x_off, const void* x_on, int64_t M, int64_t K,
                                    int64_t N, const void* W, const void* A, const void* B,
                                    int64_t r, float s, void* y_off, void* y_on, int out_dtype,
                                    void* workspace, size_t workspace_bytes, int algo,
                                    void* stream) {
  return lora_linear_impl(x_off, x_on, M, K, N, W, A, B, r, s, y_off, y_on, out_dtype, workspace,
                          workspace_bytes, algo, stream);
}

hydra_status hydra_dual_linear(const void* x_off, const void* x_on, int64_t M, int64_t K,
                               int64_t N, const void* W, const void* u, const void* B, int64_t r,
                               void* y_off, void* y_on, int out_dtype, int algo, void* stream) {
  return lora_linear_impl(x_off, x_on, M, K, N, W, nullptr, B, r, 1.0f, y_off, y_on, out_dtype,
                          const_cast<void*>(u), hydra_lora_linear_workspace_size(M, r), algo,
                          stream, true);
}

hydra_status hydra_skinny_linear(const void* x, int64_t M, int64_t K, int64_t N, const void* W,
                                 const void* u, int64_t u_row0, int64_t u_rows, const void* B,
                                 int64_t r, void* y, int out_dtype, int tile_n, int split_k,
                                 void* stream) {
  if (x == nullptr || W == nullptr || y == nullptr) return HYDRA_ERR_NULL;
  if (out_dtype != HYDRA_BF16 && out_dtype != HYDRA_F32) return HYDRA_ERR_RANGE;
  if (M < 0 || M > 128 || K < 8 || N < 16 || K >= (1LL << 31) || N >= (1LL << 31) || N % 16 != 0)
    return HYDRA_ERR_SHAPE;
  if (K % 8 != 0) return HYDRA_ERR_ALIGN;
  if (r < 0 || r > 256) return HYDRA_ERR_SHAPE;
  if (r > 0) {
    if (u == nullptr || B == nullptr) return HYDRA_ERR_NULL;
    if (r % 8 != 0) return HYDRA_ERR_ALIGN;
    if (u_rows < 1 || u_row0 < 0 || u_row0 + u_rows > M) return HYDRA_ERR_SHAPE;
    if (!aligned16(u) || !aligned16(B)) return HYDRA_ERR_ALIGN;
  }
  if (!aligned16(x) || !aligned16(W) || !aligned16(y)) return HYDRA_ERR_ALIGN;
  if (tile_n < 0 || tile_n > 256 || tile_n % 16 != 0) return HYDRA_ERR_RANGE;
  if (split_k < 0 || split_k > 8 || split_k > (K + 63) / 64) return HYDRA_ERR_RANGE;
  if (M == 0) return HYDRA_OK;
  int* err = hydra::device_error_word();
  if (err == nullptr) return HYDRA_ERR_CUDA;
  hydra::SkinnyArgs a;
  a.x = x;
  a.M = M;
  a.K = K;
  a.N = N;
  a.W = W;
  a.u = r > 0 ? u : nullptr;
  a.u_row0 = r > 0 ? u_row0 : 0;
  a.u_rows = r > 0 ? u_rows : 0;
  a.B = r > 0 ? B : nullptr;
  a.r = r;
  a.y = y;
  a.out_f32 = out_dtype == HYDRA_F32 ? 1 : 0;
  a.bn = tile_n;
  a.ks = split_k;
  a.err = err;
  return hydra::launch_skinny_gemm_tc(a, static_cast<cudaStream_t>(stream)) == 0 ? HYDRA_OK
                                                                                : HYDRA_ERR_CUDA;
}

hydra_status hydra_dual_linear_ex(const void* x_off, const void* x_on, int64_t M, int64_t K,
                                  int64_t N, const void* W, const void* u, const void* B,
                                  int64_t r, void* y_off, void* y_on, int out_dtype, int epilogue,
                                  void* stream) {
  return lora_linear_impl(x_off, x_on, M, K, N, W, nullptr, B, r, 1.0f, y_off, y_on, out_dtype,
                          const_cast<void*>(u), hydra_lora_linear_workspace_size(M, r), 1, stream,
                          true, epilogue);
}

hydra_status hydra_dual_linear_rope(const void* x_off, const void* x_on, int64_t M, int64_t K,
                                    int64_t N, const void* W, const void* u, const void* B,
                                    int64_t r, void* y_off, void* y_on, int64_t P,
                                    int64_t rope_cols, int64_t head_dim, const float* rope_table,
                                    void* stream) {
  const RopeArgs rope{P, rope_cols, head_dim, rope_table};
  return lora_linear_impl(x_off, x_on, M, K, N, W, nullptr, B, r, 1.0f, y_off, y_on, HYDRA_BF16,
                          const_cast<void*>(u), hydra_lora_linear_workspace_size(M, r), 1, stream,
                          true, kEpiRope, &rope);
}

size_t hydra_lora_linear_tri_workspace_size(int64_t M, int64_t r) {
  if (M <= 0 || r <= 0) return 0;
  return 2 * round_up(static_cast<size_t>(M) * static_cast<size_t>(r) * 2, 256);
}

hydra_status hydra_lora_linear_tri(const void* x_off, const void* x_act, const void* x_crit,
                                   int64_t M, int64_t K, int64_t N, const void* W,
                                   const void* A_act, const void* B_act, const void* A_crit,
                                   const void* B_crit, int64_t r, float s, void* y_off,
                                   void* y_act, void* y_crit, int out_dtype, void* workspace,
                                   size_t workspace_bytes, void* stream) {
  if (x_off == nullptr || x_act == nullptr || x_crit == nullptr || W == nullptr)
    return HYDRA_ERR_NULL;
  if (y_off == nullptr && y_act == nullptr && y_crit == nullptr) return HYDRA_ERR_NULL;
  if (out_dtype != HYDRA_BF16 && out_dtype != HYDRA_F32) return HYDRA_ERR_RANGE;
  if (M < 0 || K < 8 || N < 8 || M >= (1LL << 31) || K >= (1LL << 31) || N >= (1LL << 31))
    return HYDRA_ERR_SHAPE;
  if (K % 8 != 0 || N % 8 != 0) return HYDRA_ERR_ALIGN;
  if (r < 0 || r > 256) return HYDRA_ERR_SHAPE;
  if (r > 0 && r % 8 != 0) return HYDRA_ERR_ALIGN;
  if (!aligned16(x_off) || !aligned16(x_act) || !aligned16(x_crit) || !aligned16(W) ||
      !aligned16(y_off) || !aligned16(y_act) || !aligned16(y_crit))
    return HYDRA_ERR_ALIGN;
  const bool lora_a = r > 0 && y_act != nullptr, lora_c = r > 0 && y_crit != nullptr;
  if ((lora_a && (A_act == nullptr || B_act == nullptr)) ||
      (lora_c && (A_crit == nullptr || B_crit == nullptr)))
    return HYDRA_ERR_NULL;
  if ((lora_a && (!aligned16(A_act) || !aligned16(B_act))) ||
      (lora_c && (!aligned16(A_crit) || !aligned16(B_crit))))
    return HYDRA_ERR_ALIGN;
  if (lora_a || lora_c) {
    if (workspace == nullptr) return HYDRA_ERR_WORKSPACE;
    if (!aligned16(workspace)) return HYDRA_ERR_ALIGN;
    if (workspace_bytes < hydra_lora_linear_tri_workspace_size(M, r)) return HYDRA_ERR_WORKSPACE;
  }
  if (M == 0) return HYDRA_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int* err = hydra::device_error_word();
  if (err == nullptr) return HYDRA_ERR_CUDA;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  void* u_a = ws;
  void* u_c = lora_a || lora_c ? ws + round_up(static_cast<size_t>(M) * r * 2, 256) : nullptr;
  if (lora_a && hydra::launch_lora_down(x_act, M, K, A_act, r, s, u_a, st) != 0) return HYDRA_ERR_CUDA;
  if (lora_c && hydra::launch_lora_down(x_crit, M, K, A_crit, r, s, u_c, st) != 0) return HYDRA_ERR_CUDA;
  hydra::GemmArgs g;
  g.x_off = x_off;
  g.x_on = x_act;
  g.x_crit = x_crit;
  g.M = M;
  g.K = K;
  g.N = N;
  g.W = W;
  g.u = lora_a ? u_a : nullptr;
  g.B = lora_a ? B_act : nullptr;
  g.u_crit = lora_c ? u_c : nullptr;
  g.B_crit = lora_c ? B_crit : nullptr;
  g.r = (lora_a || lora_c) ? r : 0;
  g.shared_x = false;
  g.y_off = y_off;
  g.y_on = y_act;
  g.y_crit = y_crit;
  g.out_f32 = out_dtype == HYDRA_F32 ? 1 : 0;
  g.err = err;
  return hydra::launch_dual_lora_gemm_tc(g, st) == 0 ? HYDRA_OK : HYDRA_ERR_CUDA;
}

size_t hydra_lm_head_logprobs_workspace_size(int64_t S, int64_t L, int64_t V, int64_t r) {
  if (S < 0 || L < 0 || V < 1 || r < 0) return 0;
  const size_t rows = static_cast<size_t>(S) * static_cast<size_t>(L);
  const size_t nt = static_cast<size_t>((V + 255) / 256);
  return round_up(2 * rows * nt * 8, 256) + round_up(2 * rows * 4, 256) +
         round_up(rows * static_cast<size_t>(r) * 2, 256);
}

hydra_status hydra_lm_head_logprobs(const void* h_off, const void* h_on, int64_t S, int64_t L,
                                    int64_t d, int64_t V, const void* W, const void* A,
                                    const void* B, int64_t r, float s, const int32_t* ids,
                                    const int32_t* lengths, const float* seq_score, float beta,
                                    float* logp_actor, float* logp_ref, float* reward_tok,
                                    float* lse_actor, float* lse_ref, void* workspace,
                                    size_t workspace_bytes, void* stream) {
  if (h_off == nullptr || W == nullptr || ids == nullptr || logp_actor == nullptr ||
      logp_ref == nullptr || reward_tok == nullptr || workspace == nullptr)
    return HYDRA_ERR_NULL;
  if (S < 0 || L < 0 || d < 8 || V < 8 || r < 0 || r > 256) return HYDRA_ERR_SHAPE;
  if (S * L >= (1LL << 31) || d >= (1LL << 31) || V >= (1LL << 31)) return HYDRA_ERR_SHAPE;
  if (d % 8 != 0 || V % 8 != 0 || r % 8 != 0) return HYDRA_ERR_ALIGN;
  const bool shared_x = (h_on == nullptr || h_on == h_off);
  if (r > 0 && (A == nullptr || B == nullptr)) return HYDRA_ERR_NULL;
  if (!aligned16(h_off) || (!shared_x && !aligned16(h_on)) || !aligned16(W) ||
      !aligned16(workspace) || (r > 0 && (!aligned16(A) || !aligned16(B))))
    return HYDRA_ERR_ALIGN;
  if (workspace_bytes < hydra_lm_head_logprobs_workspace_size(S, L, V, r)) return HYDRA_ERR_WORKSPACE;
  const int64_t M = S * L;
  if (M == 0) return HYDRA_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int* err = hydra::device_error_word();
  if (err == nullptr) return HYDRA_ERR_CUDA;
  // workspace: partials of both heads, sampled-token logits of both heads, u
  const size_t nt = static_cast<size_t>((V + 255) / 256);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  float2* part = reinterpret_cast<float2*>(ws);
  float* tgt = reinterpret_cast<float*>(ws + round_up(2 * static_cast<size_t>(M) * nt * 8, 256));
  void* u = ws + round_up(2 * static_cast<size_t>(M) * nt * 8, 256) +
            round_up(2 * static_cast<size_t>(M) * 4, 256);
  const void* xo = shared_x ? h_off : h_on;
  if (r > 0 && hydra::launch_lora_down(xo, M, d, A, r, s, u, st) != 0) return HYDRA_ERR_CUDA;
  hydra::GemmArgs g;
  g.x_off = h_off;
  g.x_on = xo;
  g.M = M;
  g.K = d;
  g.N = V;
  g.W = W;
  g.u = r > 0 ? u : nullptr;
  g.B = r > 0 ? B : nullptr;
  g.r = r;
  g.shared_x = shared_x;
  g.y_off = part;                                  // reference head (LoRA off)
  g.y_on = part + static_cast<size_t>(M) * nt;     // actor head (LoRA on)
  g.out_f32 = 1;
  g.err = err;
  g.epi = 4;
  g.lsm_target = tgt;
  g.lsm_ids = ids;
  g.lsm_L = L;
  g.lsm_ids_ld = L;
  g.lsm_ids_off = 0;
  if (hydra::launch_dual_lora_gemm_tc(g, st) != 0) return HYDRA_ERR_CUDA;
  return hydra::launch_lse_combine(part, part + static_cast<size_t>(M) * nt, static_cast<int64_t>(nt),
                                   tgt, tgt + M, S, L, V, ids, L, lengths, seq_score, beta,
                                   logp_actor, logp_ref, reward_tok, lse_actor, lse_ref, err, st) == 0
             ? HYDRA_OK
             : HYDRA_ERR_CUDA;
}

hydra_status hydra_rope_table(int64_t P, int64_t head_dim, float theta, float* table,
                              void* stream) {
  if (table == nullptr) return HYDRA_ERR_NULL;
  if (P < 0 || head_dim < 2 || head_dim % 2 != 0) return HYDRA_ERR_SHAPE;
  if (!(theta > 0.f)) return HYDRA_ERR_RANGE;
  if (!aligned16(table)) return HYDRA_ERR_ALIGN;
  return hydra::launch_rope_table(P, head_dim, theta, table, static_cast<cudaStream_t>(stream)) == 0
             ? HYDRA_OK
             : HYDRA_ERR_CUDA;
}

hydra_status hydra_token_logprobs_kl(const void* logits_actor, const void* logits_ref,
                                     int logits_dtype, int64_t S, int64_t L, int64_t V, int64_t ld,
                                     const int32_t* ids, const int32_t* lengths,
                                     const float* seq_score, float beta, float* logp_actor,
                                     float* logp_ref, float* reward_tok, float* lse_actor,
                                     float* lse_ref, void* stream) {
  if (logits_dtype != HYDRA_F32 && logits_dtype != HYDRA_BF16) return HYDRA_ERR_RANGE;
  if (S < 0 || L < 0 || V < 1 || V >= (1LL << 31) || ld < V || S * L >= (1LL << 31))
    return HYDRA_ERR_SHAPE;
  if (S == 0 || L == 0) return HYDRA_OK;
  if (logits_actor == nullptr || logits_ref == nullptr || ids == nullptr ||
      logp_actor == nullptr || logp_ref == nullptr || reward_tok == nullptr)
    return HYDRA_ERR_NULL;
  int* err = hydra::device_error_word();
  if (err == nullptr) return HYDRA_ERR_CUDA;
  return hydra::launch_token_logprobs_kl(logits_actor, logits_ref, logits_dtype == HYDRA_BF16, S, L,
                                         V, ld, ids, L, lengths, seq_score, beta, logp_actor, logp_ref,
                                         reward_tok, lse_actor, lse_ref, err,
                                         static_cast<cudaStream_t>(stream)) == 0
             ? HYDRA_OK
             : HYDRA_ERR_CUDA;
}

hydra_status ppo_gae(const float* rewards, const float* values, const int32_t* lengths, int64_t S,
                     int64_t L, float gamma, float lam, float* advantages, float* returns,
                     void* stream) {
  if (S < 0 || L < 0 || L > hydra::kGaeMaxL || S * L >= (1LL << 40) || S >= (1LL << 31))
    return HYDRA_ERR_SHAPE;
  if (S == 0 || L == 0) return HYDRA_OK;
  if (rewards == nullptr || values == nullptr || advantages == nullptr || returns == nullptr)
    return HYDRA_ERR_NULL;
  int* err = hydra::device_error_word();
  if (err == nullptr) return HYDRA_ERR_CUDA;
  return hydra::launch_gae(rewards, values, lengths, S, L, gamma, lam, advantages, returns, err,
                           static_cast<cudaStream_t>(stream)) == 0
             ? HYDRA_OK
             : HYDRA_ERR_CUDA;
}

static bool ppo_shape_ok(int64_t S, int64_t L) {
  return S >= 0 && L >= 0 && S < (1LL << 31) && L < (1LL << 31) && S * L < (1LL << 31);
}

size_t hydra_ppo_workspace_size(void) { return hydra::ppo_loss_workspace_bytes(); }

hydra_status hydra_ppo_adv_moments(const float* advantages, const int32_t* lengths, int64_t S,
                                   int64_t L, double* moments, void* workspace,
                                   size_t workspace_bytes, void* stream) {
  if (!ppo_shape_ok(S, L)) return HYDRA_ERR_SHAPE;
  if (moments == nullptr || (S * L > 0 && advantages == nullptr)) return HYDRA_ERR_NULL;
  if (workspace == nullptr || workspace_bytes < hydra::ppo_loss_workspace_bytes() ||
      reinterpret_cast<uintptr_t>(workspace) % 16 != 0)
    return HYDRA_ERR_WORKSPACE;
  int* err = hydra::device_error_word();
  if (err == nullptr) return HYDRA_ERR_CUDA;
  return hydra::launch_ppo_adv_moments(advantages, lengths, S, L, moments, workspace, err,
                                       static_cast<cudaStream_t>(stream)) == 0
             ? HYDRA_OK
             : HYDRA_ERR_CUDA;
}

hydra_status hydra_ppo_loss(const float* logp_new, const float* logp_old, const float* advantages,
                            const float* returns, const float* values, const int32_t* lengths,
                            int64_t S, int64_t L, float clip_eps, int whiten,
                            const double* adv_moments, float* grad_logp, float* grad_values,
                            double* stats, void* workspace, size_t workspace_bytes,
                            void* stream) {
  if (!ppo_shape_ok(S, L)) return HYDRA_ERR_SHAPE;
  if (!(clip_eps >= 0.f && clip_eps < 1.f) || (whiten != 0 && whiten != 1)) return HYDRA_ERR_RANGE;
  if (stats == nullptr) return HYDRA_ERR_NULL;
  if (S * L > 0 && (logp_new == nullptr || logp_old == nullptr || advantages == nullptr ||
                    returns == nullptr || values == nullptr || grad_logp == nullptr ||
                    grad_values == nullptr))
    return HYDRA_ERR_NULL;
  if (workspace == nullptr || workspace_bytes < hydra::ppo_loss_workspace_bytes() ||
      reinterpret_cast<uintptr_t>(workspace) % 16 != 0)
    return HYDRA_ERR_WORKSPACE;
  int* err = hydra::device_error_word();
  if (err == nullptr) return HYDRA_ERR_CUDA;
  return hydra::launch_ppo_loss(logp_new, logp_old, advantages, returns, values, lengths, S, L,
                                clip_eps, whiten != 0, adv_moments, grad_logp, grad_values, stats,
                                workspace, err, static_cast<cudaStream_t>(stream)) == 0
             ? HYDRA_OK
             : HYDRA_ERR_CUDA;
}

hydra_status hydra_ppo_merge_moments(const double* moments, int64_t k, double* out) {
  if (k < 0) return HYDRA_ERR_SHAPE;
  if (out == nullptr || (k > 0 && moments == nullptr)) return HYDRA_ERR_NULL;
  double n = 0.0, mean = 0.0, m2 = 0.0;
  for (int64_t i = 0; i < k; ++i) {
    const double nb = moments[3 * i], mb = moments[3 * i + 1], m2b = moments[3 * i + 2];
    if (!(nb >= 0.0) || !(m2b >= 0.0)) return HYDRA_ERR_RANGE;
    const double nn = n + nb;
    if (nn == 0.0) continue;
    const double d = mb - mean;
    const double f = nb / nn;
    mean += d * f;
    m2 += m2b + d * d * n * f;
    n = nn;
  }
  out[0] = n;
  out[1] = mean;
  out[2] = m2;
  return HYDRA_OK;
}

}  // extern "C"
