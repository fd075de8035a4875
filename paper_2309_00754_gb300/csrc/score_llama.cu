// C-ABI of the Llama decoder pieces and the native host driver of the full J-Hydra scoring
// pass (Algorithm 1 scoring steps; §3 Dynamic LoRA and J-Hydra-PPO: one frozen base, the
// LoRA-off stream gives the reference policy and the reward model, the LoRA-on stream the
// actor and the critic). Both streams' rows are stacked so every kernel covers both in one
// launch and each projection's W tiles are fetched from HBM once.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>
#include <vector>

#include "../../include/hydra.h"
#include "kernels.h"

namespace {

// ---------------------------------------------------------------- kernel-class timing
// When enabled, hydra_score_llama brackets every launch with CUDA events recorded on the
// call's stream; hydra_profile_collect sums the elapsed times per kernel class. Events come
// from a pool that grows on demand and is reused after each collect.
struct Profiler {
  bool on = false;
  std::vector<cudaEvent_t> pool;
  size_t used = 0;
  std::vector<int> cls;  // class of event pair i (events 2i, 2i + 1)
  std::mutex mu;
} g_prof;

cudaEvent_t prof_event() {
  if (g_prof.used == g_prof.pool.size()) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    g_prof.pool.push_back(e);
  }
  return g_prof.pool[g_prof.used++];
}

struct ProfScope {
  cudaStream_t st;
  bool active;
  ProfScope(int c, cudaStream_t s) : st(s), active(g_prof.on) {
    if (!active) return;
    cudaEvent_t e = prof_event();
    if (e == nullptr) {
      active = false;
      return;
    }
    g_prof.cls.push_back(c);
    cudaEventRecord(e, st);
  }
  ~ProfScope() {
    if (!active) return;
    cudaEvent_t e = prof_event();
    if (e != nullptr) cudaEventRecord(e, st);
  }
};

inline bool a16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline size_t up256(size_t v) { return (v + 255) / 256 * 256; }
inline hydra_status rc(int r) { return r == 0 ? HYDRA_OK : HYDRA_ERR_CUDA; }

// Workspace layout of the full pass, in bytes from the workspace base.
struct PassLayout {
  size_t h, a, qkv, attn, m, u, fin, part, tgt, sc, rope, total;
};

// ns stacked streams: 2 (J-Hydra: off, on) or 3 (Hydra-PPO: off, actor, critic)
PassLayout layout(const hydra_llama_config& c, int64_t S, int ns = 2) {
  const size_t P = static_cast<size_t>(c.prompt_len + c.response_len);
  const size_t T = static_cast<size_t>(S) * P;
  const size_t R = static_cast<size_t>(ns) * T;
  const size_t d = static_cast<size_t>(c.d_model), F = static_cast<size_t>(c.ffn);
  const size_t SL = static_cast<size_t>(S) * static_cast<size_t>(c.response_len);
  PassLayout L;
  size_t o = 0;
  L.h = o;      o += up256(R * d * 4);
  L.a = o;      o += up256(R * d * 2);
  L.qkv = o;    o += up256(R * 3 * d * 2);
  L.attn = o;   o += up256(R * d * 2);
  L.m = o;      o += up256(R * F * 2);
  L.u = o;      o += up256((ns - 1) * T * 2 * static_cast<size_t>(c.lora_rank) * 2);
  L.fin = o;    o += up256(static_cast<size_t>(ns) * SL * d * 2);
  // LM head: per-(row, 256-column tile) log-softmax partials and sampled-token logits of both
  // heads (the logits themselves never reach memory)
  L.part = o;   o += up256(2 * SL * static_cast<size_t>((c.vocab + 255) / 256) * 8);
  L.tgt = o;    o += up256(2 * SL * 4);
  L.sc = o;     o += up256(static_cast<size_t>(S) * 4);
  L.rope = o;   o += up256(P * static_cast<size_t>(c.head_dim / 2) * 8);
  L.total = o;
  return L;
}

bool valid_config(const hydra_llama_config* c) {
  if (c == nullptr) return false;
  if (c->n_layers < 1 || c->head_dim != 128 || c->n_heads < 1) return false;
  if (c->d_model != c->n_heads * c->head_dim) return false;
  if (c->ffn < 128 || c->ffn % 128 != 0 || c->vocab < 8 || c->vocab % 8 != 0) return false;
  if (c->lora_rank < 8 || c->lora_rank > 128 || c->lora_rank % 8 != 0) return false;
  if (c->prompt_len < 1 || c->response_len < 1 || !(c->rope_theta > 0.f)) return false;
  if (c->response_len > hydra::kGaeMaxL) return false;
  return true;
}

// stacked linear of ns streams: rows [0, T) of x are the off stream, [T, 2T) the on
// (actor) stream and, when ns == 3, [2T, 3T) the critic stream with its own LoRA set
// (A2, B2; u2 receives its down-projection)
// epi: tcgen05 epilogue; y is [ns T, N] (store, rotary), [ns T, N/2] bf16 (SwiGLU) or the
// fp32 residual stream [ns T, N] (residual add); rope: rotary arguments of epi == kStackEpiRope
int stacked_linear_impl(int prof_class, const void* x, int64_t T, int64_t K, int64_t N,
                        const void* W, const void* A, const void* B, int64_t r, float s, void* u,
                        void* y, bool f32, int* err, cudaStream_t st, int epi,
                        const hydra::StackRope* rope, int ns, const void* A2, const void* B2,
                        void* u2) {
  const size_t xs = static_cast<size_t>(T) * K * 2;
  const size_t ys = epi == HYDRA_EPI_SWIGLU    ? static_cast<size_t>(T) * (N / 2) * 2
                    : epi == HYDRA_EPI_RESIDUAL ? static_cast<size_t>(T) * N * 4
                                                : static_cast<size_t>(T) * N * (f32 ? 4 : 2);
  const void* x_off = x;
  const void* x_on = static_cast<const uint8_t*>(x) + xs;
  const void* x_crit = static_cast<const uint8_t*>(x) + 2 * xs;
  if (r > 0) {
    ProfScope ps(HYDRA_PROF_LORA_DOWN, st);
    int e = hydra::launch_lora_down(x_on, T, K, A, r, s, u, st);
    if (e == 0 && ns == 3) e = hydra::launch_lora_down(x_crit, T, K, A2, r, s, u2, st);
    if (e != 0) return e;
  }
  ProfScope ps(prof_class, st);
  hydra::GemmArgs g;
  g.x_off = x_off;
  g.x_on = x_on;
  g.M = T;
  g.K = K;
  g.N = N;
  g.W = W;
  g.u = r > 0 ? u : nullptr;
  g.B = r > 0 ? B : nullptr;
  g.r = r;
  g.shared_x = false;
  g.y_off = y;
  g.y_on = static_cast<uint8_t*>(y) + ys;
  if (ns == 3) {
    g.x_crit = x_crit;
    g.u_crit = r > 0 ? u2 : nullptr;
    g.B_crit = r > 0 ? B2 : nullptr;
    g.y_crit = static_cast<uint8_t*>(y) + 2 * ys;
  }
  g.out_f32 = f32 ? 1 : 0;
  g.err = err;
  g.epi = epi;
  if (rope != nullptr) {
    g.rope_P = rope->P;
    g.rope_cols = rope->cols;
    g.rope_table = rope->table;
  }
  return hydra::launch_dual_lora_gemm_tc(g, st);
}

}  // namespace

namespace hydra {
int stacked_linear(int prof_class, const void* x, int64_t T, int64_t K, int64_t N, const void* W,
                   const void* A, const void* B, int64_t r, float s, void* u, void* y, bool f32,
                   int* err, cudaStream_t st, int epi, const StackRope* rope, int ns,
                   const void* A2, const void* B2, void* u2) {
  return stacked_linear_impl(prof_class, x, T, K, N, W, A, B, r, s, u, y, f32, err, st, epi, rope,
                             ns, A2, B2, u2);
}
}  // namespace hydra

extern "C" {

hydra_status hydra_embed(const void* table, int64_t V, int64_t d, const int32_t* ids, int64_t T,
                         int copies, float* h, void* stream) {
  if (table == nullptr || ids == nullptr || h == nullptr) return HYDRA_ERR_NULL;
  if (V < 1 || d < 8 || T < 0 || copies < 1 || copies > 2) return HYDRA_ERR_SHAPE;
  if (d % 8 != 0 || !a16(table) || !a16(h)) return HYDRA_ERR_ALIGN;
  int* err = hydra::device_error_word();
  if (err == nullptr) return HYDRA_ERR_CUDA;
  return rc(hydra::launch_embed(table, V, d, ids, T, copies, h, err,
                                static_cast<cudaStream_t>(stream)));
}

hydra_status hydra_rmsnorm(const float* x, const void* w, int64_t rows, int64_t d, float eps,
                           int64_t g_out, int64_t g_in, int64_t off, void* y, void* stream) {
  if (x == nullptr || w == nullptr || y == nullptr) return HYDRA_ERR_NULL;
  if (rows < 0 || d < 8 || g_out < 1 || g_in < 0 || off < 0) return HYDRA_ERR_SHAPE;
  if (d % 8 != 0 || !a16(x) || !a16(w) || !a16(y)) return HYDRA_ERR_ALIGN;
  hydra::RowMap m{g_out, g_in, off};
  return rc(hydra::launch_rmsnorm(x, w, rows, d, eps, m, y, static_cast<cudaStream_t>(stream)));
}

hydra_status hydra_rope(void* qkv, int64_t R, int64_t ld, int64_t d, int64_t head_dim, int64_t P,
                        float theta, void* stream) {
  if (qkv == nullptr) return HYDRA_ERR_NULL;
  if (R < 0 || P < 1 || head_dim < 4 || head_dim % 4 != 0 || d % head_dim != 0 || ld < 2 * d)
    return HYDRA_ERR_SHAPE;
  if (ld % 2 != 0 || (reinterpret_cast<uintptr_t>(qkv) & 3u) != 0) return HYDRA_ERR_ALIGN;
  if (!(theta > 0.f)) return HYDRA_ERR_RANGE;
  return rc(hydra::launch_rope(qkv, R, ld, d, head_dim, P, theta, static_cast<cudaStream_t>(stream)));
}

hydra_status hydra_causal_attention(const void* qkv, int64_t nseq, int64_t P, int64_t ld,
                                    int64_t n_heads, int64_t head_dim, void* out, int64_t ld_out,
                                    void* stream) {
  if (qkv == nullptr || out == nullptr) return HYDRA_ERR_NULL;
  if (head_dim != 128) return HYDRA_ERR_SHAPE;
  if (nseq < 0 || P < 0 || n_heads < 1 || ld < 3 * n_heads * head_dim ||
      ld_out < n_heads * head_dim)
    return HYDRA_ERR_SHAPE;
  if (ld % 8 != 0 || ld_out % 8 != 0 || !a16(qkv) || !a16(out)) return HYDRA_ERR_ALIGN;
  return rc(hydra::launch_causal_attention(qkv, nseq, P, ld, n_heads, head_dim, out, ld_out,
                                           static_cast<cudaStream_t>(stream)));
}

hydra_status hydra_swiglu(const void* gu, int64_t R, int64_t F, void* m, void* stream) {
  if (gu == nullptr || m == nullptr) return HYDRA_ERR_NULL;
  if (R < 0 || F < 8) return HYDRA_ERR_SHAPE;
  if (F % 8 != 0 || !a16(gu) || !a16(m)) return HYDRA_ERR_ALIGN;
  return rc(hydra::launch_swiglu(gu, R, F, m, static_cast<cudaStream_t>(stream)));
}

hydra_status hydra_residual_add(float* h, const void* y, int64_t n, void* stream) {
  if (h == nullptr || y == nullptr) return HYDRA_ERR_NULL;
  if (n < 0) return HYDRA_ERR_SHAPE;
  if (n % 8 != 0 || !a16(h) || !a16(y)) return HYDRA_ERR_ALIGN;
  return rc(hydra::launch_residual_add(h, y, n, static_cast<cudaStream_t>(stream)));
}

hydra_status hydra_head_dot(const void* x, int64_t d, const void* w, int64_t n, int64_t g_out,
                            int64_t g_in, int64_t off, float* out, void* stream) {
  if (x == nullptr || w == nullptr || out == nullptr) return HYDRA_ERR_NULL;
  if (n < 0 || d < 8 || g_out < 1 || g_in < 0 || off < 0) return HYDRA_ERR_SHAPE;
  if (d % 8 != 0 || !a16(x) || !a16(w)) return HYDRA_ERR_ALIGN;
  hydra::RowMap m{g_out, g_in, off};
  return rc(hydra::launch_head_dot(x, d, w, m, n, nullptr, 1, out,
                                   static_cast<cudaStream_t>(stream)));
}

hydra_status hydra_profile_enable(int on) {
  std::lock_guard<std::mutex> lock(g_prof.mu);
  g_prof.on = on != 0;
  return HYDRA_OK;
}

hydra_status hydra_profile_collect(float* ms, int64_t* launches, int reset) {
  if (ms == nullptr || launches == nullptr) return HYDRA_ERR_NULL;
  std::lock_guard<std::mutex> lock(g_prof.mu);
  for (int c = 0; c < HYDRA_PROF_CLASSES; ++c) {
    ms[c] = 0.f;
    launches[c] = 0;
  }
  for (size_t i = 0; i < g_prof.cls.size(); ++i) {
    if (2 * i + 1 >= g_prof.used) break;
    cudaEvent_t a = g_prof.pool[2 * i], b = g_prof.pool[2 * i + 1];
    if (cudaEventSynchronize(b) != cudaSuccess) return HYDRA_ERR_CUDA;
    float t = 0.f;
    if (cudaEventElapsedTime(&t, a, b) != cudaSuccess) return HYDRA_ERR_CUDA;
    ms[g_prof.cls[i]] += t;
    launches[g_prof.cls[i]] += 1;
  }
  if (reset) {
    g_prof.cls.clear();
    g_prof.used = 0;
  }
  return HYDRA_OK;
}

size_t hydra_score_llama_workspace_size(const hydra_llama_config* cfg, int64_t S) {
  if (!valid_config(cfg) || S < 0) return 0;
  return layout(*cfg, S).total;
}

// The scoring pass over ns = 2 (J-Hydra; critic == NULL) or 3 (Hydra-PPO: critic holds the
// critic's LoRA set per layer) stacked streams.
static hydra_status score_pass(const hydra_llama_config* cfg, const hydra_llama_weights* w,
                               const hydra_llama_lora* critic, const int32_t* ids,
                               const int32_t* lengths, int64_t S, void* workspace,
                               size_t workspace_bytes, float* logp_actor, float* logp_ref,
                               float* reward, float* values, float* advantages, float* returns,
                               float* score, void* stream) {
  if (cfg == nullptr || w == nullptr) return HYDRA_ERR_NULL;
  const int ns = critic != nullptr ? 3 : 2;
  if (!valid_config(cfg)) return HYDRA_ERR_SHAPE;
  if (S < 0) return HYDRA_ERR_SHAPE;
  if (S == 0) return HYDRA_OK;
  if (ids == nullptr || logp_actor == nullptr || logp_ref == nullptr || reward == nullptr ||
      values == nullptr || advantages == nullptr || returns == nullptr || score == nullptr)
    return HYDRA_ERR_NULL;
  if (w->embed == nullptr || w->layers == nullptr || w->final_norm == nullptr ||
      w->lm_head == nullptr || w->w_rm == nullptr)
    return HYDRA_ERR_NULL;
  const hydra_llama_config& c = *cfg;
  for (int64_t l = 0; l < c.n_layers; ++l) {
    const hydra_llama_layer& ly = w->layers[l];
    const void* ptrs[] = {ly.w_qkv, ly.a_qv, ly.b_qkv, ly.w_o, ly.w_gu, ly.a_gu,
                          ly.b_gu, ly.w_down, ly.a_down, ly.b_down, ly.norm_attn, ly.norm_ffn};
    for (const void* p : ptrs) {
      if (p == nullptr) return HYDRA_ERR_NULL;
      if (!a16(p)) return HYDRA_ERR_ALIGN;
    }
    if (critic != nullptr) {
      const hydra_llama_lora& cl = critic[l];
      const void* cp[] = {cl.a_qv, cl.b_qkv, cl.a_gu, cl.b_gu, cl.a_down, cl.b_down};
      for (const void* p : cp) {
        if (p == nullptr) return HYDRA_ERR_NULL;
        if (!a16(p)) return HYDRA_ERR_ALIGN;
      }
    }
  }
  const PassLayout Lo = layout(c, S, ns);
  if (workspace == nullptr) return HYDRA_ERR_WORKSPACE;
  if (!a16(workspace)) return HYDRA_ERR_ALIGN;
  if (workspace_bytes < Lo.total) return HYDRA_ERR_WORKSPACE;
  int* err = hydra::device_error_word();
  if (err == nullptr) return HYDRA_ERR_CUDA;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  std::unique_lock<std::mutex> prof_lock(g_prof.mu, std::defer_lock);
  if (g_prof.on) prof_lock.lock();

  uint8_t* ws = static_cast<uint8_t*>(workspace);
  float* h = reinterpret_cast<float*>(ws + Lo.h);
  void* a = ws + Lo.a;
  void* qkv = ws + Lo.qkv;
  void* attn = ws + Lo.attn;
  void* m = ws + Lo.m;
  void* u = ws + Lo.u;
  void* u2 = static_cast<uint8_t*>(u) + static_cast<size_t>(S) * (c.prompt_len + c.response_len) *
                                            2 * c.lora_rank * 2;  // critic stream's u
  void* fin = ws + Lo.fin;
  float2* part = reinterpret_cast<float2*>(ws + Lo.part);
  float* tgt = reinterpret_cast<float*>(ws + Lo.tgt);
  float* sc = reinterpret_cast<float*>(ws + Lo.sc);
  void* rope_table = ws + Lo.rope;

  const int64_t P = c.prompt_len + c.response_len;
  const int64_t T = S * P;
  const int64_t R = ns * T;
  const int64_t d = c.d_model, F = c.ffn, V = c.vocab, r = c.lora_rank, L = c.response_len;
  const int64_t SL = S * L;
  const float s = c.lora_scale;
  const hydra::RowMap ident{R, R, 0};
  // The last layer's output is read only on the rows the heads use: per sequence the L rows
  // that predict the response tokens (positions P0 - 1 .. P - 2; the actor's and reference
  // log-probabilities and the values) and the row of the last position P - 1 (the reward
  // score, at the last valid token). Its q/k/v projection and attention run over every
  // position (the prompt's keys and values); from the o projection on it runs on those
  // Lc = L + 1 rows of each sequence, gathered into compact buffers: per row the same
  // arithmetic, so the same bits.
  const int64_t Lc = L + 1, Tc = S * Lc;
  const bool compact = Lc < P;
  const hydra::RowMap pick{Lc, P, c.prompt_len - 1};  // compact row -> row of the full stream
  float* hc = reinterpret_cast<float*>(qkv);  // compact residual rows (qkv is free by then)
  int e = 0;
#define HY_TRY(x)                     \
  do {                                \
    if ((e = (x)) != 0) return rc(e); \
  } while (0)
#define HY_PROF(cls, x)        \
  do {                         \
    ProfScope ps_(cls, st);    \
    HY_TRY(x);                 \
  } while (0)

  HY_PROF(HYDRA_PROF_ELEMENTWISE, hydra::launch_embed(w->embed, V, d, ids, T, ns, h, err, st));
  // rotation table of the positions 0..P-1, shared by every layer's q/k/v epilogue
  HY_PROF(HYDRA_PROF_ELEMENTWISE, hydra::launch_rope_table(P, c.head_dim, c.rope_theta, rope_table, st));
  for (int64_t l = 0; l < c.n_layers; ++l) {
    const hydra_llama_layer& ly = w->layers[l];
    const hydra_llama_lora* cl = critic != nullptr ? &critic[l] : nullptr;  // critic LoRA set
    // attention block: q/k/v projection with the rotary embedding of q and k fused into the
    // epilogue
    const hydra::StackRope rope{P, 2 * d, rope_table};
    if (l == 0 && ns == 2) {
      // Both streams enter layer 0 with the same embedding rows, so their normed inputs are
      // equal: one accumulator per tile serves both outputs (x W^T drained to the off stream,
      // then the LoRA k-blocks accumulated on top for the on stream), the same bits as the
      // stacked form for half the products (§3 Dynamic LoRA: one frozen W, LoRA switched)
      HY_PROF(HYDRA_PROF_ELEMENTWISE, hydra::launch_rmsnorm(h, ly.norm_attn, T, d, c.rms_eps, ident, a, st));
      HY_PROF(HYDRA_PROF_LORA_DOWN, hydra::launch_lora_down(a, T, d, ly.a_qv, 2 * r, s, u, st));
      ProfScope ps(HYDRA_PROF_GEMM_QKV, st);
      hydra::GemmArgs g;
      g.x_off = a;
      g.x_on = a;
      g.M = T;
      g.K = d;
      g.N = 3 * d;
      g.W = ly.w_qkv;
      g.u = u;
      g.B = ly.b_qkv;
      g.r = 2 * r;
      g.shared_x = true;
      g.y_off = qkv;
      g.y_on = static_cast<uint8_t*>(qkv) + static_cast<size_t>(T) * 3 * d * 2;
      g.out_f32 = 0;
      g.err = err;
      g.epi = hydra::kStackEpiRope;
      g.rope_P = P;
      g.rope_cols = 2 * d;
      g.rope_table = rope_table;
      HY_TRY(hydra::launch_dual_lora_gemm_tc(g, st));
    } else {
      HY_PROF(HYDRA_PROF_ELEMENTWISE, hydra::launch_rmsnorm(h, ly.norm_attn, R, d, c.rms_eps, ident, a, st));
      HY_TRY(hydra::stacked_linear(HYDRA_PROF_GEMM_QKV, a, T, d, 3 * d, ly.w_qkv, ly.a_qv, ly.b_qkv, 2 * r, s, u, qkv, false,
                            err, st, hydra::kStackEpiRope, &rope, ns, cl ? cl->a_qv : nullptr, cl ? cl->b_qkv : nullptr, u2));
    }
    HY_PROF(HYDRA_PROF_ATTENTION,
            hydra::launch_causal_attention(qkv, ns * S, P, 3 * d, c.n_heads, c.head_dim, attn, d, st));
    // the rows this layer computes from here on: all, or the compact rows of the last layer
    // (its attention output gathered into `a`, its residual rows into `hc`)
    const bool last_c = compact && l == c.n_layers - 1;
    const int64_t Tl = last_c ? Tc : T;
    const void* x_o = attn;
    float* hl = h;
    void* al = a;
    if (last_c) {
      HY_PROF(HYDRA_PROF_ELEMENTWISE, hydra::launch_gather_rows(attn, ns * Tc, d * 2, pick, a, st));
      HY_PROF(HYDRA_PROF_ELEMENTWISE, hydra::launch_gather_rows(h, ns * Tc, d * 4, pick, hc, st));
      x_o = a;
      hl = hc;
      al = attn;
    }
    const hydra::RowMap ident_l{ns * Tl, ns * Tl, 0};
    // o projection added straight into the residual stream (fused epilogue)
    HY_TRY(hydra::stacked_linear(HYDRA_PROF_GEMM_O, x_o, Tl, d, d, ly.w_o, nullptr, nullptr, 0, s, u, hl, false, err, st,
                          HYDRA_EPI_RESIDUAL, nullptr, ns));
    // feed-forward block: gate/up with the SwiGLU fused into the epilogue, down added into the
    // residual stream
    HY_PROF(HYDRA_PROF_ELEMENTWISE, hydra::launch_rmsnorm(hl, ly.norm_ffn, ns * Tl, d, c.rms_eps, ident_l, al, st));
    HY_TRY(hydra::stacked_linear(HYDRA_PROF_GEMM_GU, al, Tl, d, 2 * F, ly.w_gu, ly.a_gu, ly.b_gu, 2 * r, s, u, m, false, err, st,
                          HYDRA_EPI_SWIGLU, nullptr, ns, cl ? cl->a_gu : nullptr, cl ? cl->b_gu : nullptr, u2));
    HY_TRY(hydra::stacked_linear(HYDRA_PROF_GEMM_DOWN, m, Tl, F, d, ly.w_down, ly.a_down, ly.b_down, r, s, u, hl, false, err, st,
                          HYDRA_EPI_RESIDUAL, nullptr, ns, cl ? cl->a_down : nullptr, cl ? cl->b_down : nullptr, u2));
  }
  // final norm on the rows that predict response tokens: row P0 - 1 + t of each sequence (row
  // t of its compact rows)
  const float* hf = compact ? hc : h;
  const hydra::RowMap resp = compact ? hydra::RowMap{L, Lc, 0} : hydra::RowMap{L, P, c.prompt_len - 1};
  HY_PROF(HYDRA_PROF_ELEMENTWISE, hydra::launch_rmsnorm(hf, w->final_norm, ns * SL, d, c.rms_eps, resp, fin, st));
  // LM head of both streams with the log-softmax reduced in the GEMM epilogue
  const int64_t nt = (V + 255) / 256;
  const int32_t* resp_ids = ids + c.prompt_len;  // token of response row s * L + t: ids[s * P + P0 + t]
  {
    ProfScope ps(HYDRA_PROF_GEMM_LMHEAD, st);
    hydra::GemmArgs g;
    g.x_off = fin;
    g.x_on = static_cast<const uint8_t*>(fin) + static_cast<size_t>(SL) * d * 2;
    g.M = SL;
    g.K = d;
    g.N = V;
    g.W = w->lm_head;
    g.r = 0;
    g.shared_x = false;
    g.y_off = part;                                // reference head (LoRA off)
    g.y_on = part + static_cast<size_t>(SL) * nt;  // actor head (LoRA on)
    g.out_f32 = 1;
    g.err = err;
    g.epi = 4;
    g.lsm_target = tgt;
    g.lsm_ids = resp_ids;
    g.lsm_L = L;
    g.lsm_ids_ld = P;
    g.lsm_ids_off = 0;
    HY_TRY(hydra::launch_dual_lora_gemm_tc(g, st));
  }
  // reward-model score on the LoRA-off stream at the last valid token; values on the
  // LoRA-on stream (the same head: r_phi = LO(V))
  // (position P0 + len - 1: compact row len of its sequence)
  HY_PROF(HYDRA_PROF_HEADS, hydra::launch_seq_score(hf, w->final_norm, w->w_rm, d, c.rms_eps,
                                                    lengths, S, L, compact ? Lc : P,
                                                    compact ? 1 : c.prompt_len, sc, st));
  // values from the last stream: the on stream (J-Hydra) or the critic stream (Hydra-PPO)
  const void* fin_on = static_cast<uint8_t*>(fin) + static_cast<size_t>(ns - 1) * SL * d * 2;
  const hydra::RowMap dense{SL, SL, 0};
  HY_PROF(HYDRA_PROF_HEADS, hydra::launch_head_dot(fin_on, d, w->w_rm, dense, SL, lengths, L, values, st));
  HY_PROF(HYDRA_PROF_LOGPROBS,
          hydra::launch_lse_combine(part, part + static_cast<size_t>(SL) * nt, nt, tgt, tgt + SL, S, L, V,
                                    resp_ids, P, lengths, sc, c.beta, logp_actor, logp_ref, reward,
                                    nullptr, nullptr, err, st));
  HY_PROF(HYDRA_PROF_GAE, hydra::launch_gae(reward, values, lengths, S, L, c.gamma, c.lam,
                                            advantages, returns, err, st));
  if (cudaMemcpyAsync(score, sc, static_cast<size_t>(S) * 4, cudaMemcpyDeviceToDevice, st) !=
      cudaSuccess)
    return HYDRA_ERR_CUDA;
#undef HY_TRY
#undef HY_PROF
  return HYDRA_OK;
}

hydra_status hydra_score_llama(const hydra_llama_config* cfg, const hydra_llama_weights* w,
                               const int32_t* ids, const int32_t* lengths, int64_t S,
                               void* workspace, size_t workspace_bytes, float* logp_actor,
                               float* logp_ref, float* reward, float* values, float* advantages,
                               float* returns, float* score, void* stream) {
  return score_pass(cfg, w, nullptr, ids, lengths, S, workspace, workspace_bytes, logp_actor,
                    logp_ref, reward, values, advantages, returns, score, stream);
}

size_t hydra_score_llama_hydra_workspace_size(const hydra_llama_config* cfg, int64_t S) {
  if (!valid_config(cfg) || S < 0) return 0;
  return layout(*cfg, S, 3).total;
}

hydra_status hydra_score_llama_hydra(const hydra_llama_config* cfg, const hydra_llama_weights* w,
                                     const hydra_llama_lora* critic, const int32_t* ids,
                                     const int32_t* lengths, int64_t S, void* workspace,
                                     size_t workspace_bytes, float* logp_actor, float* logp_ref,
                                     float* reward, float* values, float* advantages,
                                     float* returns, float* score, void* stream) {
  if (critic == nullptr) return HYDRA_ERR_NULL;
  return score_pass(cfg, w, critic, ids, lengths, S, workspace, workspace_bytes, logp_actor,
                    logp_ref, reward, values, advantages, returns, score, stream);
}

}  // extern "C"
