// Fused vocabulary-wide log-softmax + gather for the actor and reference heads, and the
// KL-penalised per-token reward (Algorithms 1 and 2: the LoRA-off model gives the reward and
// the reference log-probabilities, from which the advantages follow; §2 ratio
// r(theta) needs the actor's log-probabilities; Appendix B: KL coefficient beta).
//
// One CTA per token row streams both heads' logits once with 128-bit loads, keeping a
// running (max, sum of exp) per thread (online normaliser of Milakov & Gimelshein 2018),
// merges the partial pairs with warp shuffles and one shared-memory step, and emits
//   logp_h  = z_h[id] - lse_h,   lse_h = log sum_v exp z_h[v]     (h = actor, ref)
//   reward  = -beta (logp_actor - logp_ref) + [t == len - 1] score
// Rows at or beyond their sequence's length are not read and are written as 0.
#include <float.h>

#include "common.cuh"
#include "kernels.h"

namespace hydra {
namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ void online4(float& m, float& s, float a, float b, float c, float d) {
  const float mx = fmaxf(fmaxf(a, b), fmaxf(c, d));
  if (mx > m) {
    s *= __expf(m - mx);
    m = mx;
  }
  s += __expf(a - m) + __expf(b - m) + __expf(c - m) + __expf(d - m);
}

__device__ __forceinline__ void online1(float& m, float& s, float a) {
  if (a > m) {
    s *= __expf(m - a);
    m = a;
  }
  s += __expf(a - m);
}

__device__ __forceinline__ void merge(float& m, float& s, float m2, float s2) {
  const float mn = fmaxf(m, m2);
  s = s * __expf(m - mn) + s2 * __expf(m2 - mn);
  m = mn;
}

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(__nv_bfloat16 v) { return __bfloat162float(v); }

template <typename T>
struct Vec;
template <>
struct Vec<float> {
  static constexpr int kElems = 4;
  __device__ static __forceinline__ void consume(const float* p, int i, float& m, float& s) {
    const float4 v = __ldcs(reinterpret_cast<const float4*>(p) + i);
    online4(m, s, v.x, v.y, v.z, v.w);
  }
};
template <>
struct Vec<__nv_bfloat16> {
  static constexpr int kElems = 8;
  __device__ static __forceinline__ void consume(const __nv_bfloat16* p, int i, float& m,
                                                 float& s) {
    const uint4 v = __ldcs(reinterpret_cast<const uint4*>(p) + i);
    const float2 a = unpack_bf16x2(v.x), b = unpack_bf16x2(v.y);
    const float2 c = unpack_bf16x2(v.z), d = unpack_bf16x2(v.w);
    online4(m, s, a.x, a.y, b.x, b.y);
    online4(m, s, c.x, c.y, d.x, d.y);
  }
};

template <typename T, bool kVec>
__global__ void __launch_bounds__(kThreads)
    logprobs_kl_kernel(const T* __restrict__ za, const T* __restrict__ zr, int L, int V,
                       long long ld, const int32_t* __restrict__ ids, long long ids_ld,
                       const int32_t* __restrict__ lengths, const float* __restrict__ score,
                       float beta, float* __restrict__ la, float* __restrict__ lr,
                       float* __restrict__ rew, float* __restrict__ lse_a,
                       float* __restrict__ lse_r, int* err) {
  const long long row = blockIdx.x;
  const int s = static_cast<int>(row / L);
  const int t = static_cast<int>(row - static_cast<long long>(s) * L);
  int n = lengths ? lengths[s] : L;
  if (n < 0 || n > L) {
    if (threadIdx.x == 0) record_error(err, kDevBadLength);
    n = n < 0 ? 0 : L;
  }
  if (t >= n) {
    if (threadIdx.x == 0) {
      la[row] = 0.f;
      lr[row] = 0.f;
      rew[row] = 0.f;
      if (lse_a) lse_a[row] = 0.f;
      if (lse_r) lse_r[row] = 0.f;
    }
    return;
  }
  const T* pa = za + row * ld;
  const T* pr = zr + row * ld;
  float ma = -FLT_MAX, sa = 0.f, mr = -FLT_MAX, sr = 0.f;
  int tail_start = 0;
  if (kVec) {
    constexpr int E = Vec<T>::kElems;
    const int nv = V / E;
    int i = threadIdx.x;
    // four independent 16-byte loads per head in flight per thread
    for (; i + 3 * kThreads < nv; i += 4 * kThreads) {
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        Vec<T>::consume(pa, i + u * kThreads, ma, sa);
        Vec<T>::consume(pr, i + u * kThreads, mr, sr);
      }
    }
    for (; i < nv; i += kThreads) {
      Vec<T>::consume(pa, i, ma, sa);
      Vec<T>::consume(pr, i, mr, sr);
    }
    tail_start = nv * E;
  }
  for (int v = tail_start + threadIdx.x; v < V; v += kThreads) {
    online1(ma, sa, to_f(pa[v]));
    online1(mr, sr, to_f(pr[v]));
  }

#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    merge(ma, sa, __shfl_xor_sync(0xffffffffu, ma, off), __shfl_xor_sync(0xffffffffu, sa, off));
    merge(mr, sr, __shfl_xor_sync(0xffffffffu, mr, off), __shfl_xor_sync(0xffffffffu, sr, off));
  }
  __shared__ float red[4][kThreads / 32];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (lane == 0) {
    red[0][warp] = ma;
    red[1][warp] = sa;
    red[2][warp] = mr;
    red[3][warp] = sr;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < kThreads / 32; ++w) {
      merge(ma, sa, red[0][w], red[1][w]);
      merge(mr, sr, red[2][w], red[3][w]);
    }
    const float lsa = ma + logf(sa);
    const float lsr = mr + logf(sr);
    const int id = ids[static_cast<long long>(s) * ids_ld + t];
    float va, vr, rw;
    if (id < 0 || id >= V) {
      record_error(err, kDevBadTokenId);
      va = vr = rw = __int_as_float(0x7fc00000);
    } else {
      va = to_f(pa[id]) - lsa;
      vr = to_f(pr[id]) - lsr;
      rw = -beta * (va - vr);
      if (score != nullptr && t == n - 1) rw += score[s];
    }
    la[row] = va;
    lr[row] = vr;
    rew[row] = rw;
    if (lse_a) lse_a[row] = lsa;
    if (lse_r) lse_r[row] = lsr;
  }
}

template <typename T>
int launch_t(const void* za, const void* zr, int64_t S, int64_t L, int64_t V, int64_t ld,
             const int32_t* ids, int64_t ids_ld, const int32_t* lengths, const float* score, float beta, float* la,
             float* lr, float* rew, float* lse_a, float* lse_r, int* err, cudaStream_t stream) {
  const T* a = static_cast<const T*>(za);
  const T* r = static_cast<const T*>(zr);
  constexpr int E = Vec<T>::kElems;
  const bool vec = (reinterpret_cast<uintptr_t>(a) % 16 == 0) &&
                   (reinterpret_cast<uintptr_t>(r) % 16 == 0) && (ld % E == 0);
  const unsigned grid = static_cast<unsigned>(S * L);
  if (vec)
    logprobs_kl_kernel<T, true><<<grid, kThreads, 0, stream>>>(
        a, r, static_cast<int>(L), static_cast<int>(V), ld, ids, ids_ld, lengths, score, beta, la, lr, rew,
        lse_a, lse_r, err);
  else
    logprobs_kl_kernel<T, false><<<grid, kThreads, 0, stream>>>(
        a, r, static_cast<int>(L), static_cast<int>(V), ld, ids, ids_ld, lengths, score, beta, la, lr, rew,
        lse_a, lse_r, err);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

// One warp per token row: merges the row's per-tile (max, sum exp) partials of both heads,
// written by the log-softmax epilogue of the LM-head GEMM (the logits never reach memory),
// into lse_h, and emits logp_h = z_h[id] - lse_h and the reward exactly as
// logprobs_kl_kernel does. Head 0 (part0, tgt0) is the reference (LoRA off), head 1 the actor.
__global__ void __launch_bounds__(256)
    lse_combine_kernel(const float2* __restrict__ part0, const float2* __restrict__ part1,
                       int n_tiles, const float* __restrict__ tgt0, const float* __restrict__ tgt1,
                       long long rows, int L, int V, const int32_t* __restrict__ ids,
                       long long ids_ld, const int32_t* __restrict__ lengths,
                       const float* __restrict__ score, float beta, float* __restrict__ la,
                       float* __restrict__ lr, float* __restrict__ rew, float* __restrict__ lse_a,
                       float* __restrict__ lse_r, int* err) {
  const long long row = blockIdx.x * 8LL + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const int s = static_cast<int>(row / L);
  const int t = static_cast<int>(row - static_cast<long long>(s) * L);
  int n = lengths ? lengths[s] : L;
  if (n < 0 || n > L) {
    if (lane == 0) record_error(err, kDevBadLength);
    n = n < 0 ? 0 : L;
  }
  if (t >= n) {
    if (lane == 0) {
      la[row] = 0.f;
      lr[row] = 0.f;
      rew[row] = 0.f;
      if (lse_a) lse_a[row] = 0.f;
      if (lse_r) lse_r[row] = 0.f;
    }
    return;
  }
  float ma = -FLT_MAX, sa = 0.f, mr = -FLT_MAX, sr = 0.f;
  for (int k = lane; k < n_tiles; k += 32) {
    const float2 pr = part0[row * n_tiles + k], pa = part1[row * n_tiles + k];
    merge(mr, sr, pr.x, pr.y);
    merge(ma, sa, pa.x, pa.y);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    merge(ma, sa, __shfl_xor_sync(0xffffffffu, ma, off), __shfl_xor_sync(0xffffffffu, sa, off));
    merge(mr, sr, __shfl_xor_sync(0xffffffffu, mr, off), __shfl_xor_sync(0xffffffffu, sr, off));
  }
  if (lane == 0) {
    const float lsa = ma + logf(sa);
    const float lsr = mr + logf(sr);
    const int id = ids[static_cast<long long>(s) * ids_ld + t];
    float va, vr, rw;
    if (id < 0 || id >= V) {
      record_error(err, kDevBadTokenId);
      va = vr = rw = __int_as_float(0x7fc00000);
    } else {
      va = tgt1[row] - lsa;
      vr = tgt0[row] - lsr;
      rw = -beta * (va - vr);
      if (score != nullptr && t == n - 1) rw += score[s];
    }
    la[row] = va;
    lr[row] = vr;
    rew[row] = rw;
    if (lse_a) lse_a[row] = lsa;
    if (lse_r) lse_r[row] = lsr;
  }
}

}  // namespace

int launch_lse_combine(const void* part_ref, const void* part_act, int64_t n_tiles,
                       const float* tgt_ref, const float* tgt_act, int64_t S, int64_t L, int64_t V,
                       const int32_t* ids, int64_t ids_ld, const int32_t* lengths,
                       const float* score, float beta, float* la, float* lr, float* rew,
                       float* lse_a, float* lse_r, int* err, cudaStream_t stream) {
  const int64_t rows = S * L;
  if (rows == 0) return 0;
  lse_combine_kernel<<<static_cast<unsigned>((rows + 7) / 8), 256, 0, stream>>>(
      static_cast<const float2*>(part_ref), static_cast<const float2*>(part_act),
      static_cast<int>(n_tiles), tgt_ref, tgt_act, rows, static_cast<int>(L), static_cast<int>(V),
      ids, ids_ld, lengths, score, beta, la, lr, rew, lse_a, lse_r, err);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

int launch_token_logprobs_kl(const void* za, const void* zr, int bf16_logits, int64_t S, int64_t L,
                             int64_t V, int64_t ld, const int32_t* ids, int64_t ids_ld,
                             const int32_t* lengths, const float* score, float beta, float* la,
                             float* lr, float* rew, float* lse_a, float* lse_r, int* err,
                             cudaStream_t stream) {
  if (S == 0 || L == 0) return 0;
  if (bf16_logits)
    return launch_t<__nv_bfloat16>(za, zr, S, L, V, ld, ids, ids_ld, lengths, score, beta, la, lr, rew,
                                   lse_a, lse_r, err, stream);
  return launch_t<float>(za, zr, S, L, V, ld, ids, ids_ld, lengths, score, beta, la, lr, rew, lse_a, lse_r,
                         err, stream);
}

}  // namespace hydra
