// Native host driver of the KV-cached generation loop (Algorithms 1 and 2: the actor, the
// LoRA-on model, generates each sequence for T steps; J-Hydra-PPO retains the critic head's
// values while generating). The LoRA-off stream runs beside the actor in every step: decode
// is bound by reading W, and the dual-output GEMV serves both streams' rows from one read
// of each W tile, so the reference log-probability of every drawn token comes with the draw.
//
// Prefill: the prompt of both streams through the tcgen05 layer loop of the scoring pass
// (rotary, SwiGLU and residual epilogues), with each layer's rotated keys and values copied
// into the cache. Decode step (R = 2 S rows: off rows then on rows): embed the last drawn
// token, per layer [residual + RMSNorm + q/v LoRA down] -> q/k/v GEMV -> [rotary + cache
// append + attention over the cache] -> o GEMV -> [residual + RMSNorm + gate/up LoRA down]
// -> gate/up GEMV -> [SwiGLU + down LoRA down] -> down GEMV; then [residual + final RMSNorm],
// the LM-head GEMV (fp32 logits) and the draw. The norm brackets are thread-block-cluster
// kernels.
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/hydra.h"
#include "kernels.h"

namespace {

inline bool a16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline size_t up256(size_t v) { return (v + 255) / 256 * 256; }
inline hydra_status rc(int r) { return r == 0 ? HYDRA_OK : HYDRA_ERR_CUDA; }

// Up to 8 sequences both streams' rows fit one dual GEMV (16 rows); larger batches (up to 64
// sequences, 128 rows per stream-pair tile) run the decode projections on the tcgen05 GEMM,
// which also reads each W tile once.
constexpr int64_t kMaxGenSeqs = 64;

struct GenLayout {
  size_t h, a, qkv, attn, m, u;                                       // prefill, 2 S P0 rows
  size_t cache;                                                       // K/V of every layer
  size_t hd, ad, qkvd, attnd, yd, gud, md, ud, find, logits, cur, step, rope;  // decode
  size_t total;
};

GenLayout gen_layout(const hydra_llama_config& c, int64_t S) {
  const size_t P0 = static_cast<size_t>(c.prompt_len);
  const size_t Pmax = P0 + static_cast<size_t>(c.response_len);
  const size_t R = 2 * static_cast<size_t>(S);
  const size_t Rp = R * P0;
  const size_t d = static_cast<size_t>(c.d_model), F = static_cast<size_t>(c.ffn);
  const size_t r2 = 2 * static_cast<size_t>(c.lora_rank);
  GenLayout L;
  size_t o = 0;
  L.h = o;      o += up256(Rp * d * 4);
  L.a = o;      o += up256(Rp * d * 2);
  L.qkv = o;    o += up256(Rp * 3 * d * 2);
  L.attn = o;   o += up256(Rp * d * 2);
  L.m = o;      o += up256(Rp * F * 2);
  L.u = o;      o += up256(static_cast<size_t>(S) * P0 * r2 * 2);
  L.cache = o;  o += up256(static_cast<size_t>(c.n_layers) * 2 * R * Pmax * d * 2);
  L.hd = o;     o += up256(R * d * 4);
  L.ad = o;     o += up256(R * d * 2);
  L.qkvd = o;   o += up256(R * 3 * d * 2);
  L.attnd = o;  o += up256(R * d * 2);
  L.yd = o;     o += up256(R * d * 2);
  L.gud = o;    o += up256(R * 2 * F * 2);
  L.md = o;     o += up256(R * F * 2);
  L.ud = o;     o += up256(static_cast<size_t>(S) * r2 * 2);
  L.find = o;   o += up256(R * d * 2);
  L.logits = o; o += up256(R * static_cast<size_t>(c.vocab) * 4);
  L.cur = o;    o += up256(static_cast<size_t>(S) * 4);
  L.step = o;   o += 256;
  L.rope = o;   o += up256(Pmax * static_cast<size_t>(c.head_dim / 2) * 8);
  L.total = o;
  return L;
}

bool gen_config_ok(const hydra_llama_config* c) {
  if (c == nullptr) return false;
  if (c->n_layers < 1 || c->head_dim != 128 || c->n_heads < 1) return false;
  if (c->d_model != c->n_heads * c->head_dim) return false;
  if (c->ffn < 128 || c->ffn % 128 != 0 || c->vocab < 8 || c->vocab % 8 != 0) return false;
  if (c->lora_rank < 8 || c->lora_rank > 128 || c->lora_rank % 8 != 0) return false;
  if (c->prompt_len < 1 || c->response_len < 1 || !(c->rope_theta > 0.f)) return false;
  // the decode attention keeps one score per cached position in shared memory
  if (hydra::decode_attention_smem(c->prompt_len + c->response_len) > 200 * 1024) return false;
  return true;
}

// y = [x_off; x_on] W^T (+ u B^T on the on rows; u [S, r] = s x_on A^T, already computed by
// the fused row kernel that produced x) for S rows per stream; y [2 S, N] bf16 or fp32 (off
// rows first). Kernel by rows and width, as measured on GB300 (7B decode step, both streams):
//  * up to 8 rows: the dual-output GEMV (4 sequences: 3.73 ms per step against 3.97 ms with
//    the split-K kernel on the wide projections);
//  * 9 to 16 rows: the split-K tcgen05 kernel for outputs of 8192 columns and more, the GEMV
//    for the narrower ones (8 sequences: 3.93 ms, against 4.48 ms all-GEMV and 4.13 ms
//    all-split-K);
//  * above 16 rows: the split-K kernel over both streams' rows in one tile (the CTA-tile GEMM
//    when N is not a multiple of 16).
int decode_linear(const void* x, int64_t S, int64_t K, int64_t N, const void* W, const void* B,
                  int64_t r, const void* u, void* y, bool f32, int* err, cudaStream_t st) {
  const int64_t rows = 2 * S;
  const bool split_k = rows > hydra::kGemvMaxRows || (rows > 8 && N >= 8192);
  if (split_k && hydra::skinny_gemm_supported(rows, K, N, r)) {
    hydra::SkinnyArgs a;
    a.x = x;
    a.M = 2 * S;
    a.K = K;
    a.N = N;
    a.W = W;
    a.u = r > 0 ? u : nullptr;
    a.u_row0 = r > 0 ? S : 0;
    a.u_rows = r > 0 ? S : 0;
    a.B = r > 0 ? B : nullptr;
    a.r = r;
    a.y = y;
    a.out_f32 = f32 ? 1 : 0;
    a.bn = 0;
    a.ks = 0;
    a.err = err;
    return hydra::launch_skinny_gemm_tc(a, st);
  }
  hydra::GemmArgs g;
  g.x_off = x;
  g.x_on = static_cast<const uint8_t*>(x) + static_cast<size_t>(S) * K * 2;
  g.M = S;
  g.K = K;
  g.N = N;
  g.W = W;
  g.u = r > 0 ? u : nullptr;
  g.B = r > 0 ? B : nullptr;
  g.r = r;
  g.shared_x = false;
  g.y_off = y;
  g.y_on = static_cast<uint8_t*>(y) + static_cast<size_t>(S) * N * (f32 ? 4 : 2);
  g.out_f32 = f32 ? 1 : 0;
  g.err = err;
  return 2 * S <= hydra::kGemvMaxRows ? hydra::launch_dual_lora_gemv(g, st)
                                       : hydra::launch_dual_lora_gemm_tc(g, st);
}

}  // namespace

extern "C" {

size_t hydra_generate_llama_workspace_size(const hydra_llama_config* cfg, int64_t S) {
  if (!gen_config_ok(cfg) || S < 1 || S > kMaxGenSeqs) return 0;
  return gen_layout(*cfg, S).total;
}

hydra_status hydra_generate_llama(const hydra_llama_config* cfg, const hydra_llama_weights* w,
                                  const int32_t* prompt_ids, int64_t S, int64_t n_steps,
                                  const float* gumbel, void* workspace, size_t workspace_bytes,
                                  int32_t* tokens, float* logp_actor, float* logp_ref,
                                  float* values, float* score, void* stream) {
  if (cfg == nullptr || w == nullptr) return HYDRA_ERR_NULL;
  if (!gen_config_ok(cfg)) return HYDRA_ERR_SHAPE;
  const hydra_llama_config& c = *cfg;
  if (S < 1 || S > kMaxGenSeqs || n_steps < 1 || n_steps > c.response_len) return HYDRA_ERR_SHAPE;
  if (prompt_ids == nullptr || tokens == nullptr || logp_actor == nullptr ||
      logp_ref == nullptr || values == nullptr)
    return HYDRA_ERR_NULL;
  if (w->embed == nullptr || w->layers == nullptr || w->final_norm == nullptr ||
      w->lm_head == nullptr || w->w_rm == nullptr)
    return HYDRA_ERR_NULL;
  for (int64_t l = 0; l < c.n_layers; ++l) {
    const hydra_llama_layer& ly = w->layers[l];
    const void* ptrs[] = {ly.w_qkv, ly.a_qv, ly.b_qkv, ly.w_o, ly.w_gu, ly.a_gu,
                          ly.b_gu, ly.w_down, ly.a_down, ly.b_down, ly.norm_attn, ly.norm_ffn};
    for (const void* p : ptrs) {
      if (p == nullptr) return HYDRA_ERR_NULL;
      if (!a16(p)) return HYDRA_ERR_ALIGN;
    }
  }
  const GenLayout Lo = gen_layout(c, S);
  if (workspace == nullptr) return HYDRA_ERR_WORKSPACE;
  if (!a16(workspace)) return HYDRA_ERR_ALIGN;
  if (workspace_bytes < Lo.total) return HYDRA_ERR_WORKSPACE;
  int* err = hydra::device_error_word();
  if (err == nullptr) return HYDRA_ERR_CUDA;
  cudaStream_t st = static_cast<cudaStream_t>(stream);

  uint8_t* ws = static_cast<uint8_t*>(workspace);
  const int64_t P0 = c.prompt_len, Pmax = c.prompt_len + c.response_len;
  const int64_t d = c.d_model, F = c.ffn, V = c.vocab, r = c.lora_rank, H = c.n_heads;
  const int64_t R = 2 * S, T = S * P0;
  const float s = c.lora_scale;
  const size_t layer_kv = static_cast<size_t>(R) * H * Pmax * 128 * 2;  // bytes of K (or V)
  float* h = reinterpret_cast<float*>(ws + Lo.h);
  void* a = ws + Lo.a;
  void* qkv = ws + Lo.qkv;
  void* attn = ws + Lo.attn;
  void* m = ws + Lo.m;
  void* u = ws + Lo.u;
  uint8_t* cache = ws + Lo.cache;
  float* hd = reinterpret_cast<float*>(ws + Lo.hd);
  void* ad = ws + Lo.ad;
  void* qkvd = ws + Lo.qkvd;
  void* attnd = ws + Lo.attnd;
  void* yd = ws + Lo.yd;
  void* gud = ws + Lo.gud;
  void* md = ws + Lo.md;
  void* ud = ws + Lo.ud;
  void* find = ws + Lo.find;
  float* logits = reinterpret_cast<float*>(ws + Lo.logits);
  int32_t* cur = reinterpret_cast<int32_t*>(ws + Lo.cur);
  int* step = reinterpret_cast<int*>(ws + Lo.step);
  void* rope_table = ws + Lo.rope;
  auto kcache = [&](int64_t l) { return cache + 2 * layer_kv * static_cast<size_t>(l); };
  auto vcache = [&](int64_t l) { return cache + 2 * layer_kv * static_cast<size_t>(l) + layer_kv; };

  int e = 0;
#define HY_TRY(x)                     \
  do {                                \
    if ((e = (x)) != 0) return rc(e); \
  } while (0)

  if (cudaMemsetAsync(step, 0, sizeof(int), st) != cudaSuccess) return HYDRA_ERR_CUDA;
  HY_TRY(hydra::launch_rope_table(Pmax, c.head_dim, c.rope_theta, rope_table, st));

  // ---- prefill: the prompt of both streams, keys and values into the cache
  const hydra::RowMap ident{R * P0, R * P0, 0};
  HY_TRY(hydra::launch_embed(w->embed, V, d, prompt_ids, T, 2, h, err, st));
  for (int64_t l = 0; l < c.n_layers; ++l) {
    const hydra_llama_layer& ly = w->layers[l];
    HY_TRY(hydra::launch_rmsnorm(h, ly.norm_attn, R * P0, d, c.rms_eps, ident, a, st));
    const hydra::StackRope rope{P0, 2 * d, rope_table};
    HY_TRY(hydra::stacked_linear(HYDRA_PROF_GEMM_QKV, a, T, d, 3 * d, ly.w_qkv, ly.a_qv, ly.b_qkv,
                                 2 * r, s, u, qkv, false, err, st, hydra::kStackEpiRope, &rope));
    HY_TRY(hydra::launch_kv_store_prefill(qkv, R, P0, 3 * d, d, H, Pmax, kcache(l), vcache(l), st));
    HY_TRY(hydra::launch_causal_attention(qkv, R, P0, 3 * d, H, c.head_dim, attn, d, st));
    HY_TRY(hydra::stacked_linear(HYDRA_PROF_GEMM_O, attn, T, d, d, ly.w_o, nullptr, nullptr, 0, s,
                                 u, h, false, err, st, HYDRA_EPI_RESIDUAL));
    HY_TRY(hydra::launch_rmsnorm(h, ly.norm_ffn, R * P0, d, c.rms_eps, ident, a, st));
    HY_TRY(hydra::stacked_linear(HYDRA_PROF_GEMM_GU, a, T, d, 2 * F, ly.w_gu, ly.a_gu, ly.b_gu,
                                 2 * r, s, u, m, false, err, st, HYDRA_EPI_SWIGLU));
    HY_TRY(hydra::stacked_linear(HYDRA_PROF_GEMM_DOWN, m, T, F, d, ly.w_down, ly.a_down,
                                 ly.b_down, r, s, u, h, false, err, st, HYDRA_EPI_RESIDUAL));
  }
  // the last prompt position of every row: rows i P0 + P0 - 1
  const hydra::RowMap last{1, P0, P0 - 1};
  HY_TRY(hydra::launch_rmsnorm(h, w->final_norm, R, d, c.rms_eps, last, find, st));

  // one decode pass of the last drawn token (cur), ending in the final-normed rows find. Its
  // embedding launch advances the device-side step counter to the number of tokens drawn, so
  // the pass runs at position P0 + step - 1. Eight launches per layer: the residual add, the
  // RMSNorm and the next projection's LoRA down-projection share one cluster kernel, as do
  // the SwiGLU and the down projection's LoRA down-projection.
  auto decode_layers = [&]() -> int {
    int x = hydra::launch_embed(w->embed, V, d, cur, S, 2, hd, err, st, step);
    const void* resid = nullptr;  // the previous layer's down projection, added into h
    for (int64_t l = 0; l < c.n_layers && x == 0; ++l) {
      const hydra_llama_layer& ly = w->layers[l];
      if ((x = hydra::launch_row_norm_lora(hd, resid, ly.norm_attn, R, d, c.rms_eps, ad, S, ly.a_qv,
                                           2 * r, s, ud, st)) != 0)
        break;
      if ((x = decode_linear(ad, S, d, 3 * d, ly.w_qkv, ly.b_qkv, 2 * r, ud, qkvd, false, err, st)) != 0)
        break;
      if ((x = hydra::launch_decode_attention(qkvd, R, 3 * d, d, H, rope_table, kcache(l),
                                              vcache(l), P0, step, Pmax, attnd, d, st)) != 0)
        break;
      if ((x = decode_linear(attnd, S, d, d, ly.w_o, nullptr, 0, ud, yd, false, err, st)) != 0) break;
      if ((x = hydra::launch_row_norm_lora(hd, yd, ly.norm_ffn, R, d, c.rms_eps, ad, S, ly.a_gu,
                                           2 * r, s, ud, st)) != 0)
        break;
      if ((x = decode_linear(ad, S, d, 2 * F, ly.w_gu, ly.b_gu, 2 * r, ud, gud, false, err, st)) != 0)
        break;
      if ((x = hydra::launch_swiglu_lora(gud, R, F, md, S, ly.a_down, r, s, ud, st)) != 0) break;
      if ((x = decode_linear(md, S, F, d, ly.w_down, ly.b_down, r, ud, yd, false, err, st)) != 0) break;
      resid = yd;
    }
    if (x == 0)
      x = hydra::launch_row_norm_lora(hd, resid, w->final_norm, R, d, c.rms_eps, find, S, nullptr, 0,
                                      s, nullptr, st);
    return x;
  };
  // the LM head on both streams' final rows and the draw of step *step (the count so far)
  auto draw = [&]() -> int {
    int x = decode_linear(find, S, d, V, w->lm_head, nullptr, 0, nullptr, logits, true, err, st);
    if (x == 0)
      x = hydra::launch_sample_tokens(logits, S, V, gumbel, find, d, w->w_rm, step, n_steps, tokens,
                                      logp_actor, logp_ref, values, cur, st);
    return x;
  };

  HY_TRY(draw());
  for (int64_t t = 1; t < n_steps; ++t) {
    HY_TRY(decode_layers());
    HY_TRY(draw());
  }
  if (score != nullptr) {
    // the reward model (LoRA off) on the state after the last drawn token
    HY_TRY(decode_layers());
    const hydra::RowMap dense{R, R, 0};
    HY_TRY(hydra::launch_head_dot(find, d, w->w_rm, dense, S, nullptr, 1, score, st));
  }
#undef HY_TRY
  return HYDRA_OK;
}

}  // extern "C"
