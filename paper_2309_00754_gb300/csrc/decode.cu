// Kernels of the KV-cached generation loop (Algorithms 1 and 2: the actor samples each
// sequence for T steps; J-Hydra-PPO keeps the critic head's value of every step). The decode
// step runs the R = 2 S stacked rows of the LoRA-off and LoRA-on streams of S sequences; the
// projections are the dual-output GEMV (up to 16 rows) or the split-K tcgen05 linear, the rest
// is here:
//   kv_store_prefill   the prompt's rotated keys and its values into the cache
//   row_norm_lora      (8-CTA clusters) residual add + RMSNorm + the next projection's LoRA
//                      down-projection
//   swiglu_lora        (8-CTA clusters) SwiGLU + the down projection's LoRA down-projection
//                      (row_norm_lora also in a grouped form, several rows per cluster,
//                      above 96 rows)
//   decode_attention   rotary embedding of the new token's q and k, its k and v appended to
//                      the cache, then one query row per (head, row) against the cached
//                      positions 0..pos
//   sample_tokens      per sequence: log-softmax of both heads, the Gumbel-max draw from the
//                      actor's logits, both log-probabilities of the drawn token, the value
// The step counter lives in device memory: kernels read the position from it rather than
// from their launch arguments, so every step issues identical launches.
// Cache layout per layer: K [R][H][Pmax][Dh] then V [R][H][Pmax][Dh], bf16, row i = stream
// * S + sequence.
#include <algorithm>
#include <utility>

#include "common.cuh"
#include "kernels.h"

namespace hydra {
namespace {

constexpr int kDh = 128;  // head_dim of every decoder in this library

__global__ void kv_store_prefill_kernel(const __nv_bfloat16* __restrict__ qkv, int P0, int ld,
                                        int d, int H, int Pmax, __nv_bfloat16* __restrict__ ck,
                                        __nv_bfloat16* __restrict__ cv) {
  // block = one prompt row (i, p); 8 bf16 per thread step over the k and v blocks
  const long long row = blockIdx.x;
  const int i = static_cast<int>(row / P0), p = static_cast<int>(row % P0);
  const __nv_bfloat16* src = qkv + static_cast<size_t>(row) * ld;
  for (int e = threadIdx.x * 8; e < 2 * d; e += blockDim.x * 8) {
    const int kv = e >= d ? 1 : 0;
    const int c = e - kv * d;
    const int h = c / kDh, j = c % kDh;
    const uint4 v = *reinterpret_cast<const uint4*>(src + d + e);
    __nv_bfloat16* dst = (kv ? cv : ck) + ((static_cast<size_t>(i) * H + h) * Pmax + p) * kDh + j;
    *reinterpret_cast<uint4*>(dst) = v;
  }
}

constexpr int kAttnThreads = 256;
constexpr int kAttnWarps = kAttnThreads / 32;

__device__ __forceinline__ float block_max(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  const int warp = threadIdx.x >> 5;
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[warp] = v;
  __syncthreads();
  v = red[0];
  for (int w = 1; w < static_cast<int>(blockDim.x >> 5); ++w) v = fmaxf(v, red[w]);
  return v;
}

__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int warp = threadIdx.x >> 5;
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[warp] = v;
  __syncthreads();
  v = 0.f;
  for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) v += red[w];
  return v;
}

// One block per (head, row): the new token's rotary and cache append for this head, then the
// scores of the npos = pos + 1 cached keys into shared memory
// (groups of 8 lanes per key, 32 bytes each, reduced by shuffles), the softmax over them,
// then the weighted sum of the values (lane = 4 output dimensions, warps split positions).
// Each iteration loads its own keys: for large batches, bound by HBM bandwidth (small batches
// take decode_attention_1p_kernel below).
__global__ void __launch_bounds__(kAttnThreads)
    decode_attention_kernel(const __nv_bfloat16* __restrict__ qkv, int ld, int d, int H,
                            const float2* __restrict__ table, __nv_bfloat16* __restrict__ ck,
                            __nv_bfloat16* __restrict__ cv, int P0,
                            const int* __restrict__ step, int Pmax, float scale,
                            __nv_bfloat16* __restrict__ out, int ld_out) {
  extern __shared__ float sc[];  // [Pmax] scores, then [kAttnWarps][kDh] partial outputs
  __shared__ float red[kAttnWarps];
  __shared__ __align__(16) __nv_bfloat16 qs[kDh];  // this head's rotated query
  pdl_wait();
  pdl_launch_dependents();
  const int h = blockIdx.x, i = blockIdx.y;
  const int pos = P0 + *step - 1;
  if (pos < 0 || pos >= Pmax) return;  // the host keeps every step inside the cache
  const int npos = pos + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __nv_bfloat16* K = ck + (static_cast<size_t>(i) * H + h) * Pmax * kDh;
  __nv_bfloat16* Vc = cv + (static_cast<size_t>(i) * H + h) * Pmax * kDh;
  {
    // the new token: rotary embedding of this head's q (into shared memory) and k (into the
    // cache at pos), and its v copied into the cache; the same explicit roundings as the
    // prefill's rotary, from the same table
    constexpr int half = kDh / 2;
    const __nv_bfloat16* row = qkv + static_cast<size_t>(i) * ld;
    if (threadIdx.x < 2 * half) {
      const int j = threadIdx.x & (half - 1), blk = threadIdx.x / half;  // 0: q, 1: k
      const float2 cs = table[static_cast<size_t>(pos) * half + j];
      const __nv_bfloat16* x = row + blk * d + h * kDh;
      const float x1 = __bfloat162float(x[j]), x2 = __bfloat162float(x[j + half]);
      const __nv_bfloat16 o1 = __float2bfloat16_rn(__fsub_rn(__fmul_rn(x1, cs.x), __fmul_rn(x2, cs.y)));
      const __nv_bfloat16 o2 = __float2bfloat16_rn(__fadd_rn(__fmul_rn(x1, cs.y), __fmul_rn(x2, cs.x)));
      __nv_bfloat16* dst = blk == 0 ? qs : K + static_cast<size_t>(pos) * kDh;
      dst[j] = o1;
      dst[j + half] = o2;
    } else if (threadIdx.x < 2 * half + kDh / 8) {
      const int e = 8 * (threadIdx.x - 2 * half);
      *reinterpret_cast<uint4*>(Vc + static_cast<size_t>(pos) * kDh + e) =
          *reinterpret_cast<const uint4*>(row + 2 * d + h * kDh + e);
    }
  }
  __syncthreads();  // q in shared memory, the new k and v visible to the whole block
  const int g = lane >> 3, sub = lane & 7;
  float qf[16];
  {
    const uint4 a = *reinterpret_cast<const uint4*>(qs + 16 * sub);
    const uint4 b = *reinterpret_cast<const uint4*>(qs + 16 * sub + 8);
    const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float2 f = unpack_bf16x2(w[k]);
      qf[2 * k] = f.x * scale;
      qf[2 * k + 1] = f.y * scale;
    }
  }
  // warp-uniform trip count: all 32 lanes reach the shuffles. Each 8-lane group takes two
  // keys per iteration, both loaded before either is reduced.
  constexpr int kKeysPerIter = 2 * 4 * kAttnWarps;
  auto load_keys = [&](int base, uint4 (&kk)[4]) {
    const int q0 = base + g, q1 = base + 4 * kAttnWarps + g;
    kk[0] = kk[1] = kk[2] = kk[3] = make_uint4(0u, 0u, 0u, 0u);
    if (q0 < npos) {
      const __nv_bfloat16* kr = K + static_cast<size_t>(q0) * kDh + 16 * sub;
      kk[0] = __ldcs(reinterpret_cast<const uint4*>(kr));
      kk[1] = __ldcs(reinterpret_cast<const uint4*>(kr + 8));
    }
    if (q1 < npos) {
      const __nv_bfloat16* kr = K + static_cast<size_t>(q1) * kDh + 16 * sub;
      kk[2] = __ldcs(reinterpret_cast<const uint4*>(kr));
      kk[3] = __ldcs(reinterpret_cast<const uint4*>(kr + 8));
    }
  };
  uint4 cur[4];
  for (int base = warp * 4; base < npos; base += kKeysPerIter) {
    const int p0 = base + g, p1 = base + 4 * kAttnWarps + g;
    load_keys(base, cur);
    const uint4 a0 = cur[0], b0 = cur[1], a1 = cur[2], b1 = cur[3];
    const uint32_t w0[8] = {a0.x, a0.y, a0.z, a0.w, b0.x, b0.y, b0.z, b0.w};
    const uint32_t w1[8] = {a1.x, a1.y, a1.z, a1.w, b1.x, b1.y, b1.z, b1.w};
    float acc0 = 0.f, acc1 = 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float2 f0 = unpack_bf16x2(w0[k]), f1 = unpack_bf16x2(w1[k]);
      acc0 = fmaf(qf[2 * k], f0.x, acc0);
      acc0 = fmaf(qf[2 * k + 1], f0.y, acc0);
      acc1 = fmaf(qf[2 * k], f1.x, acc1);
      acc1 = fmaf(qf[2 * k + 1], f1.y, acc1);
    }
#pragma unroll
    for (int o = 1; o < 8; o <<= 1) {
      acc0 += __shfl_xor_sync(0xffffffffu, acc0, o);
      acc1 += __shfl_xor_sync(0xffffffffu, acc1, o);
    }
    if (sub == 0 && p0 < npos) sc[p0] = acc0;
    if (sub == 0 && p1 < npos) sc[p1] = acc1;
  }
  __syncthreads();
  float m = -INFINITY;
  for (int p = threadIdx.x; p < npos; p += kAttnThreads) m = fmaxf(m, sc[p]);
  m = block_max(m, red);
  float l = 0.f;
  for (int p = threadIdx.x; p < npos; p += kAttnThreads) {
    const float e = expf(sc[p] - m);
    sc[p] = e;
    l += e;
  }
  l = block_sum(l, red);  // ends with a barrier: every weight is in shared memory
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 8
  for (int p = warp; p < npos; p += kAttnWarps) {
    const float wgt = sc[p];
    const uint2 v = __ldcs(reinterpret_cast<const uint2*>(Vc + static_cast<size_t>(p) * kDh + 4 * lane));
    const float2 v0 = unpack_bf16x2(v.x), v1 = unpack_bf16x2(v.y);
    acc[0] = fmaf(wgt, v0.x, acc[0]);
    acc[1] = fmaf(wgt, v0.y, acc[1]);
    acc[2] = fmaf(wgt, v1.x, acc[2]);
    acc[3] = fmaf(wgt, v1.y, acc[3]);
  }
  float* part = sc + Pmax;
#pragma unroll
  for (int k = 0; k < 4; ++k) part[warp * kDh + 4 * lane + k] = acc[k];
  __syncthreads();
  const float inv = 1.f / l;
  for (int t = threadIdx.x; t < kDh; t += kAttnThreads) {
    float o = 0.f;
#pragma unroll
    for (int w = 0; w < kAttnWarps; ++w) o += part[w * kDh + t];
    out[static_cast<size_t>(i) * ld_out + h * kDh + t] = __float2bfloat16_rn(o * inv);
  }
}


// Single-pass form for small batches: 32 groups of 8 lanes per block (lane = 16 dimensions of
// a key or value row); group G takes positions G + 32 t, two per iteration, and the K and V
// rows of the next two iterations are in flight (cp.async into a shared-memory ring) while
// this one's are reduced. Each group keeps a
// lazily rescaled running maximum (moved only when a score exceeds it by more than 2^8, as in
// the prefill's flash attention), its sum and its 16-dimension slice of the weighted values;
// the 32 partial results meet in shared memory at the end.
constexpr int kAttnGroups = kAttnThreads / 8;
constexpr int kAttnStages = 3;                          // iterations of K / V loads staged
constexpr int kAttnStageBytes = 2 * kAttnGroups * 512;  // two positions per group, K and V
constexpr uint32_t kAttnPrefetchPiece = 4096;           // bytes per L2 prefetch
__global__ void __launch_bounds__(kAttnThreads)
    decode_attention_1p_kernel(const __nv_bfloat16* __restrict__ qkv, int ld, int d, int H,
                               const float2* __restrict__ table, __nv_bfloat16* __restrict__ ck,
                               __nv_bfloat16* __restrict__ cv, int P0,
                               const int* __restrict__ step, int Pmax, float scale_log2,
                               __nv_bfloat16* __restrict__ out, int ld_out) {
  extern __shared__ float part[];  // the K / V ring; after it, [kAttnGroups][kDh] partial
                                   // outputs, then [kAttnGroups][2]
  __shared__ __align__(16) __nv_bfloat16 qs[kDh];
  const int h = blockIdx.x, i = blockIdx.y;
  __nv_bfloat16* K = ck + (static_cast<size_t>(i) * H + h) * Pmax * kDh;
  __nv_bfloat16* Vc = cv + (static_cast<size_t>(i) * H + h) * Pmax * kDh;
  {
    // The cached keys and values of earlier positions are final: this (row, head)'s stream
    // into L2 while the q/k/v projection finishes. The step counter read here may not have
    // advanced yet; a prefetch is only a hint, clamped to the cache.
    const int hint = min(max(P0 + *reinterpret_cast<const volatile int*>(step) - 1, 0), Pmax);
    const uint32_t bytes = static_cast<uint32_t>(hint) * kDh * 2;  // a multiple of 256
    const uint32_t pieces = (bytes + kAttnPrefetchPiece - 1) / kAttnPrefetchPiece;
    for (uint32_t q = threadIdx.x; q < 2 * pieces; q += kAttnThreads) {
      const bool isv = q >= pieces;
      const uint32_t off = (isv ? q - pieces : q) * kAttnPrefetchPiece;
      prefetch_l2_bulk(reinterpret_cast<const uint8_t*>(isv ? Vc : K) + off,
                       min(kAttnPrefetchPiece, bytes - off));
    }
  }
  pdl_wait();
  pdl_launch_dependents();
  const int pos = P0 + *step - 1;
  if (pos < 0 || pos >= Pmax) return;  // the host keeps every step inside the cache
  const int npos = pos + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 3, sub = lane & 7;
  const int G = warp * 4 + g;
  // rows of positions G + 32 (2 t + e), e = 0, 1: each lane copies its 32 bytes of K and of V
  // into stage t % kAttnStages of a shared-memory ring with cp.async (missing positions read
  // as zeros), so kAttnStages - 1 iterations of loads are in flight while one is reduced; a
  // lane reads back only the bytes it copied itself
  const uint32_t ring = smem_u32(part);
  auto slot = [&](int stage, int e) {
    return ring + stage * kAttnStageBytes + (e * kAttnGroups + G) * 512 + 32 * sub;
  };
  auto load = [&](int t) {
    const int stage = t % kAttnStages;
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int p = G + kAttnGroups * (2 * t + e);
      const bool ok = p < npos;
      const size_t off = static_cast<size_t>(ok ? p : 0) * kDh + 16 * sub;
      const uint32_t dst = slot(stage, e);
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst + 16 * h2),
                     "l"(K + off + 8 * h2), "r"(ok ? 16 : 0)
                     : "memory");
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst + 256 + 16 * h2),
                     "l"(Vc + off + 8 * h2), "r"(ok ? 16 : 0)
                     : "memory");
      }
    }
  };
  const int iters = (npos + 2 * kAttnGroups - 1) / (2 * kAttnGroups);  // block-uniform
  auto prologue = [&]() {
#pragma unroll
    for (int t = 0; t < kAttnStages - 1; ++t) {
      if (t < iters) load(t);
      asm volatile("cp.async.commit_group;" ::: "memory");
    }
  };
  // The first kAttnStages - 1 iterations' loads go out before the rotary and the cache append
  // when none of their positions is this step's (block-uniform); otherwise after them.
  const bool early = (kAttnStages - 1) * 2 * kAttnGroups <= pos;
  if (early) prologue();
  {
    constexpr int half = kDh / 2;
    const __nv_bfloat16* row = qkv + static_cast<size_t>(i) * ld;
    if (threadIdx.x < 2 * half) {
      const int j = threadIdx.x & (half - 1), blk = threadIdx.x / half;  // 0: q, 1: k
      const float2 cs = table[static_cast<size_t>(pos) * half + j];
      const __nv_bfloat16* x = row + blk * d + h * kDh;
      const float x1 = __bfloat162float(x[j]), x2 = __bfloat162float(x[j + half]);
      const __nv_bfloat16 o1 = __float2bfloat16_rn(__fsub_rn(__fmul_rn(x1, cs.x), __fmul_rn(x2, cs.y)));
      const __nv_bfloat16 o2 = __float2bfloat16_rn(__fadd_rn(__fmul_rn(x1, cs.y), __fmul_rn(x2, cs.x)));
      __nv_bfloat16* dst = blk == 0 ? qs : K + static_cast<size_t>(pos) * kDh;
      dst[j] = o1;
      dst[j + half] = o2;
    } else if (threadIdx.x < 2 * half + kDh / 8) {
      const int e = 8 * (threadIdx.x - 2 * half);
      *reinterpret_cast<uint4*>(Vc + static_cast<size_t>(pos) * kDh + e) =
          *reinterpret_cast<const uint4*>(row + 2 * d + h * kDh + e);
    }
  }
  __syncthreads();  // q in shared memory, the new k and v in the cache before any lane copies them
  float qf[16];
  {
    const uint4 a = *reinterpret_cast<const uint4*>(qs + 16 * sub);
    const uint4 b = *reinterpret_cast<const uint4*>(qs + 16 * sub + 8);
    const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float2 f = unpack_bf16x2(w[k]);
      qf[2 * k] = f.x * scale_log2;
      qf[2 * k + 1] = f.y * scale_log2;
    }
  }
  float acc[16];
#pragma unroll
  for (int k = 0; k < 16; ++k) acc[k] = 0.f;
  float m_ref = -INFINITY, l = 0.f;
  if (!early) prologue();
  for (int t = 0; t < iters; ++t) {
    if (t + kAttnStages - 1 < iters) load(t + kAttnStages - 1);
    asm volatile("cp.async.commit_group;" ::: "memory");
    asm volatile("cp.async.wait_group %0;" ::"n"(kAttnStages - 1) : "memory");
    const int stage = t % kAttnStages;
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int p = G + kAttnGroups * (2 * t + e);
      const uint32_t src = slot(stage, e);
      uint4 k0, k1, v0, v1;
      asm volatile("ld.shared.v4.b32 {%0,%1,%2,%3}, [%4];" : "=r"(k0.x), "=r"(k0.y), "=r"(k0.z), "=r"(k0.w) : "r"(src));
      asm volatile("ld.shared.v4.b32 {%0,%1,%2,%3}, [%4];" : "=r"(k1.x), "=r"(k1.y), "=r"(k1.z), "=r"(k1.w) : "r"(src + 16));
      const uint32_t kw[8] = {k0.x, k0.y, k0.z, k0.w, k1.x, k1.y, k1.z, k1.w};
      float sdot = 0.f;
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float2 f = unpack_bf16x2(kw[k]);
        sdot = fmaf(qf[2 * k], f.x, sdot);
        sdot = fmaf(qf[2 * k + 1], f.y, sdot);
      }
#pragma unroll
      for (int o = 1; o < 8; o <<= 1) sdot += __shfl_xor_sync(0xffffffffu, sdot, o);
      if (p < npos) {  // uniform over the 8 lanes of a group
        if (sdot > m_ref + 8.f) {
          const float corr = exp2f(m_ref - sdot);
#pragma unroll
          for (int k = 0; k < 16; ++k) acc[k] *= corr;
          l *= corr;
          m_ref = sdot;
        }
        const float wgt = exp2f(sdot - m_ref);
        l += wgt;
        asm volatile("ld.shared.v4.b32 {%0,%1,%2,%3}, [%4];" : "=r"(v0.x), "=r"(v0.y), "=r"(v0.z), "=r"(v0.w) : "r"(src + 256));
        asm volatile("ld.shared.v4.b32 {%0,%1,%2,%3}, [%4];" : "=r"(v1.x), "=r"(v1.y), "=r"(v1.z), "=r"(v1.w) : "r"(src + 272));
        const uint32_t vw[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const float2 f = unpack_bf16x2(vw[k]);
          acc[2 * k] = fmaf(wgt, f.x, acc[2 * k]);
          acc[2 * k + 1] = fmaf(wgt, f.y, acc[2 * k + 1]);
        }
      }
    }
  }
  asm volatile("cp.async.wait_group 0;" ::: "memory");
  __syncthreads();  // the ring is free before it holds the partial results
  float* ml = part + kAttnGroups * kDh;
#pragma unroll
  for (int k = 0; k < 16; ++k) part[G * kDh + 16 * sub + k] = acc[k];
  if (sub == 0) {
    ml[2 * G] = m_ref;
    ml[2 * G + 1] = l;
  }
  __syncthreads();
  if (threadIdx.x < kDh) {
    float M = -INFINITY;
#pragma unroll 8
    for (int q = 0; q < kAttnGroups; ++q) M = fmaxf(M, ml[2 * q]);
    float o = 0.f, L = 0.f;
#pragma unroll 8
    for (int q = 0; q < kAttnGroups; ++q) {
      const float f = exp2f(ml[2 * q] - M);  // 0 for a group without positions
      o = fmaf(f, part[q * kDh + threadIdx.x], o);
      L = fmaf(f, ml[2 * q + 1], L);
    }
    out[static_cast<size_t>(i) * ld_out + h * kDh + threadIdx.x] = __float2bfloat16_rn(o / L);
  }
}

// ---------------------------------------------------------------- fused row kernels
// Thread-block clusters of kCl CTAs share one row: each CTA owns a 1/kCl slice of the columns,
// partial sums meet through distributed shared memory and are added in CTA-rank order, so the
// result does not depend on timing. The one-row kernels push their partials into the CTAs
// that add them (st.shared::cluster), so one cluster barrier makes them visible and no CTA
// reads another's shared memory after it; the grouped kernels read them (ld.shared::cluster).
constexpr int kCl = 8;
constexpr int kRowThreads = 256;
constexpr int kRowWarps = kRowThreads / 32;
constexpr int kMaxR2 = 256;  // LoRA ranks of one fused down-projection (2 r for q/v, gate/up)

__device__ __forceinline__ float row_block_sum(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  float t = 0.f;
#pragma unroll
  for (int w = 0; w < kRowWarps; ++w) t += red[w];
  return t;
}

// The LoRA factor A is frozen: a CTA copies its slice A[0:r2][c0:c0+n] into shared memory
// with cp.async before it waits on the preceding kernel, so the copy overlaps that kernel's
// tail. Slices above kMaxAPrefetch bytes are read from global memory instead.
constexpr int kMaxAPrefetch = 64 * 1024;

__device__ __forceinline__ void prefetch_a_slice(const __nv_bfloat16* __restrict__ A, int K,
                                                 int c0, int n, int r2, __nv_bfloat16* As) {
  const int per_row = n / 8;  // 16-byte pieces per row (n % 8 == 0)
  for (int c = threadIdx.x; c < r2 * per_row; c += kRowThreads) {
    const int j = c / per_row, e = (c - j * per_row) * 8;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(As + j * n + e)),
                 "l"(A + static_cast<size_t>(j) * K + c0 + e)
                 : "memory");
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
}

// the cluster's CTAs have all started (the arrive at kernel start, the wait before the first
// store into another CTA's shared memory)
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
}
__device__ __forceinline__ void st_cluster_f32(float* local, uint32_t rank, float v) {
  uint32_t raddr;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(raddr) : "r"(smem_u32(local)), "r"(rank));
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(raddr), "f"(v) : "memory");
}

// Partial LoRA down-projection of this CTA's slice, pushed into rank 0's shared memory:
// recv[rank][j] = sum_e xs[e] A[j][c0 + e] for j < r2 (warps take j in turn, lanes 4 columns
// at a time); after one cluster barrier rank 0 adds the kCl partials in rank order and writes
// u = bf16(s * sum). xs holds the slice's bf16 values; As, if not NULL, the prefetched slice
// of A ([r2][n]). No CTA reads another's shared memory after the barrier, so every CTA may
// leave once it has passed it.
__device__ __forceinline__ void lora_slice_push(const float* xs, int n, int c0, int K,
                                                const __nv_bfloat16* __restrict__ A,
                                                const __nv_bfloat16* As, int r2, float s,
                                                float* recv, __nv_bfloat16* __restrict__ u_row,
                                                uint32_t rank) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int j = warp; j < r2; j += kRowWarps) {
    const __nv_bfloat16* aj = As ? As + static_cast<size_t>(j) * n : A + static_cast<size_t>(j) * K + c0;
    float acc = 0.f;
    for (int e = 4 * lane; e < n; e += 128) {
      const uint2 q = *reinterpret_cast<const uint2*>(aj + e);
      const float2 a01 = unpack_bf16x2(q.x), a23 = unpack_bf16x2(q.y);
      acc = fmaf(xs[e], a01.x, acc);
      acc = fmaf(xs[e + 1], a01.y, acc);
      acc = fmaf(xs[e + 2], a23.x, acc);
      acc = fmaf(xs[e + 3], a23.y, acc);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) st_cluster_f32(recv + static_cast<int>(rank) * kMaxR2 + j, 0, acc);
  }
  cluster_sync_all();
  if (rank == 0) {
    for (int j = threadIdx.x; j < r2; j += kRowThreads) {
      float t = 0.f;
      for (uint32_t q = 0; q < kCl; ++q) t += recv[q * kMaxR2 + j];
      u_row[j] = __float2bfloat16_rn(s * t);
    }
  }
}

__device__ __forceinline__ void wait_a_slice() {
  asm volatile("cp.async.wait_group 0;" ::: "memory");
  __syncthreads();
}

// Cluster (kCl, 1, 1) per row of h [R, d]: h += y (RESID), a = bf16(rmsnorm(h) w) and, for the
// LoRA-on rows i >= S, u[i - S] = bf16(s a A^T) (A [r2, d]; none if A is NULL). The residual
// add, the norm and the LoRA down-projection of the next projection in one launch.
template <bool RESID>
__global__ void __launch_bounds__(kRowThreads)
    row_norm_lora_kernel(float* __restrict__ h, const __nv_bfloat16* __restrict__ y,
                         const __nv_bfloat16* __restrict__ w, int d, float eps,
                         __nv_bfloat16* __restrict__ a, int S, const __nv_bfloat16* __restrict__ A,
                         int r2, float s, __nv_bfloat16* __restrict__ u) {
  extern __shared__ float xs[];  // this CTA's slice of the row, then the prefetched A slice
  __shared__ float red[kRowWarps];
  __shared__ float parts[kCl];              // every rank's sum of squares, pushed by each rank
  __shared__ float recv[kCl * kMaxR2];      // rank 0: every rank's LoRA partials
  const uint32_t rank = cluster_rank();
  const int row = blockIdx.y;
  const int n = d / kCl, c0 = static_cast<int>(rank) * n;
  const bool lora = A != nullptr && row >= S;
  cluster_arrive_relaxed();
  __nv_bfloat16* As = (lora && r2 * n * 2 <= kMaxAPrefetch) ? reinterpret_cast<__nv_bfloat16*>(xs + n)
                                                             : nullptr;
  if (As) prefetch_a_slice(A, d, c0, n, r2, As);
  pdl_wait();
  pdl_launch_dependents();
  float* hr = h + static_cast<size_t>(row) * d + c0;
  float ss = 0.f;
  for (int e = 4 * threadIdx.x; e < n; e += 4 * kRowThreads) {
    float4 v = *reinterpret_cast<const float4*>(hr + e);
    if (RESID) {
      const uint2 q = *reinterpret_cast<const uint2*>(y + static_cast<size_t>(row) * d + c0 + e);
      const float2 y01 = unpack_bf16x2(q.x), y23 = unpack_bf16x2(q.y);
      v.x += y01.x;
      v.y += y01.y;
      v.z += y23.x;
      v.w += y23.y;
      *reinterpret_cast<float4*>(hr + e) = v;
    }
    xs[e] = v.x;
    xs[e + 1] = v.y;
    xs[e + 2] = v.z;
    xs[e + 3] = v.w;
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  ss = row_block_sum(ss, red);
  cluster_wait();  // every CTA of the cluster has started
  if (threadIdx.x < kCl) st_cluster_f32(&parts[rank], threadIdx.x, ss);
  cluster_sync_all();
  float tot = 0.f;
  for (uint32_t q = 0; q < kCl; ++q) tot += parts[q];
  const float inv = rsqrtf(tot / static_cast<float>(d) + eps);
  __nv_bfloat16* ar = a + static_cast<size_t>(row) * d + c0;
  for (int e = 4 * threadIdx.x; e < n; e += 4 * kRowThreads) {
    const uint2 wq = __ldg(reinterpret_cast<const uint2*>(w + c0 + e));
    const float2 w01 = unpack_bf16x2(wq.x), w23 = unpack_bf16x2(wq.y);
    const uint32_t o0 = pack_bf16x2(xs[e] * inv * w01.x, xs[e + 1] * inv * w01.y);
    const uint32_t o1 = pack_bf16x2(xs[e + 2] * inv * w23.x, xs[e + 3] * inv * w23.y);
    *reinterpret_cast<uint2*>(ar + e) = make_uint2(o0, o1);
    const float2 b01 = unpack_bf16x2(o0), b23 = unpack_bf16x2(o1);
    xs[e] = b01.x;
    xs[e + 1] = b01.y;
    xs[e + 2] = b23.x;
    xs[e + 3] = b23.y;
  }
  if (As) wait_a_slice();
  else __syncthreads();
  if (lora)  // the same on every CTA of the cluster (one row)
    lora_slice_push(xs, n, c0, d, A, As, r2, s, recv, u + static_cast<size_t>(row - S) * r2, rank);
}

// Cluster (kCl, 1, 1) per row of gu [R, 2F] (gate/up interleaved in blocks of 128):
// m = bf16(silu(gate) up) [R, F] and, for the LoRA-on rows, u[i - S] = bf16(s m A^T)
// (A [r, F]): SwiGLU and the down projection's LoRA down-projection in one launch.
__global__ void __launch_bounds__(kRowThreads)
    swiglu_lora_kernel(const __nv_bfloat16* __restrict__ gu, int F, __nv_bfloat16* __restrict__ m,
                       int S, const __nv_bfloat16* __restrict__ A, int r, float s,
                       __nv_bfloat16* __restrict__ u) {
  extern __shared__ float xs[];  // this CTA's slice of m, then the prefetched A slice
  __shared__ float recv[kCl * kMaxR2];  // rank 0: every rank's LoRA partials
  const uint32_t rank = cluster_rank();
  const int row = blockIdx.y;
  const int n = F / kCl, c0 = static_cast<int>(rank) * n;
  const bool lora = A != nullptr && row >= S;  // the same on every CTA of the cluster
  if (lora) cluster_arrive_relaxed();
  __nv_bfloat16* As = (lora && r * n * 2 <= kMaxAPrefetch) ? reinterpret_cast<__nv_bfloat16*>(xs + n)
                                                            : nullptr;
  if (As) prefetch_a_slice(A, F, c0, n, r, As);
  pdl_wait();
  pdl_launch_dependents();
  const __nv_bfloat16* g = gu + static_cast<size_t>(row) * 2 * F;
  __nv_bfloat16* mr = m + static_cast<size_t>(row) * F + c0;
  for (int e = 4 * threadIdx.x; e < n; e += 4 * kRowThreads) {
    const int f = c0 + e;  // 4 features inside one block of 128
    const int b = f / 128, j = f % 128;
    const uint2 gq = *reinterpret_cast<const uint2*>(g + 256 * b + j);
    const uint2 uq = *reinterpret_cast<const uint2*>(g + 256 * b + 128 + j);
    const float2 g01 = unpack_bf16x2(gq.x), g23 = unpack_bf16x2(gq.y);
    const float2 u01 = unpack_bf16x2(uq.x), u23 = unpack_bf16x2(uq.y);
    const uint32_t o0 = pack_bf16x2(g01.x / (1.0f + expf(-g01.x)) * u01.x,
                                    g01.y / (1.0f + expf(-g01.y)) * u01.y);
    const uint32_t o1 = pack_bf16x2(g23.x / (1.0f + expf(-g23.x)) * u23.x,
                                    g23.y / (1.0f + expf(-g23.y)) * u23.y);
    *reinterpret_cast<uint2*>(mr + e) = make_uint2(o0, o1);
    const float2 b01 = unpack_bf16x2(o0), b23 = unpack_bf16x2(o1);
    xs[e] = b01.x;
    xs[e + 1] = b01.y;
    xs[e + 2] = b23.x;
    xs[e + 3] = b23.y;
  }
  if (As) wait_a_slice();
  else __syncthreads();
  if (lora) {
    cluster_wait();  // every CTA of the cluster has started
    lora_slice_push(xs, n, c0, F, A, As, r, s, recv, u + static_cast<size_t>(row - S) * r, rank);
  }
}

// ---------------------------------------------------------------- grouped row kernels
// For the largest decode batches: the same fused work with a cluster of kCl CTAs per group
// of up to kMaxRpc rows (each CTA still owns a 1/kCl slice of the columns). Warp w handles
// rows w, w + 8, ... of the group, so a row's sums stay inside one warp; the LoRA factor's
// slice is read once per CTA for all of the group's LoRA-on rows instead of once per row;
// the group pays three cluster barriers, as the one-row kernels once did.
// Measured on GB300 (decode step of the 7B model): groups of R / 32 rows gave 7.82 ms against
// 8.09 ms for one cluster per row at 128 rows, but 6.24 against 6.01 ms at 64 rows. A grouped
// SwiGLU kernel (slices of 1376 features per warp) was slower than one cluster per row even at
// 128 rows (14.0 against 13.0 us per launch) and is not used.
constexpr int kMaxRpc = 8;
constexpr int kGroupMinRows = 97;     // fewer rows keep one cluster per row
constexpr int kGroupRowsPerCta = 32;  // a CTA takes ceil(R / 32) rows (at most kMaxRpc)
constexpr int kRowUnroll = 4;         // loads a lane issues before it uses the first

// Partial LoRA down-projection of the group's LoRA-on rows [i0, rows) (xs [rows][n] holds this
// CTA's bf16 slices as floats): up[(i - i0) r2 + j] = sum_e xs[i][e] A[j][c0 + e], warps over
// j, lanes over e as in lora_slice; then the kCl partials of every output are added in rank
// order, the outputs spread over the cluster's threads: u[u0 + i - i0] = bf16(s * sum).
__device__ __forceinline__ void lora_group(const float* xs, int rows, int i0, int n, int c0, int K,
                                           const __nv_bfloat16* __restrict__ A,
                                           const __nv_bfloat16* As, int r2, float s, float* up,
                                           __nv_bfloat16* __restrict__ u, int u0, uint32_t rank) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int non = rows - i0;
  for (int j = warp; j < r2; j += kRowWarps) {
    const __nv_bfloat16* aj = As ? As + static_cast<size_t>(j) * n : A + static_cast<size_t>(j) * K + c0;
    float acc[kMaxRpc];
#pragma unroll
    for (int i = 0; i < kMaxRpc; ++i) acc[i] = 0.f;
    for (int e = 4 * lane; e < n; e += 128) {
      const uint2 q = *reinterpret_cast<const uint2*>(aj + e);
      const float2 a01 = unpack_bf16x2(q.x), a23 = unpack_bf16x2(q.y);
#pragma unroll
      for (int i = 0; i < kMaxRpc; ++i) {
        if (i < non) {
          const float4 x = *reinterpret_cast<const float4*>(xs + static_cast<size_t>(i0 + i) * n + e);
          acc[i] = fmaf(x.x, a01.x, acc[i]);
          acc[i] = fmaf(x.y, a01.y, acc[i]);
          acc[i] = fmaf(x.z, a23.x, acc[i]);
          acc[i] = fmaf(x.w, a23.y, acc[i]);
        }
      }
    }
#pragma unroll
    for (int i = 0; i < kMaxRpc; ++i) {
      if (i < non) {
        float v = acc[i];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane == 0) up[i * r2 + j] = v;
      }
    }
  }
  cluster_sync_all();
  for (int f = static_cast<int>(rank) * kRowThreads + threadIdx.x; f < non * r2; f += kCl * kRowThreads) {
    float t = 0.f;
    for (uint32_t q = 0; q < kCl; ++q) t += ld_cluster_f32(up + f, q);
    const int i = f / r2, j = f - i * r2;
    u[static_cast<size_t>(u0 + i) * r2 + j] = __float2bfloat16_rn(s * t);
  }
}

// Cluster (kCl, 1, 1) per group of rpc rows of h [R, d]: row_norm_lora_kernel's work.
template <bool RESID>
__global__ void __launch_bounds__(kRowThreads)
    row_norm_lora_group_kernel(float* __restrict__ h, const __nv_bfloat16* __restrict__ y,
                               const __nv_bfloat16* __restrict__ w, int R, int rpc, int d, float eps,
                               __nv_bfloat16* __restrict__ a, int S,
                               const __nv_bfloat16* __restrict__ A, int r2, float s,
                               __nv_bfloat16* __restrict__ u) {
  extern __shared__ float xs[];  // [rpc][n] slices, then up [rpc][r2], then the A slice
  __shared__ float ssq[kMaxRpc];
  const uint32_t rank = cluster_rank();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row0 = blockIdx.y * rpc;
  const int rows = min(rpc, R - row0);
  const int n = d / kCl, c0 = static_cast<int>(rank) * n;
  const int i0 = min(rows, max(0, S - row0));  // first LoRA-on row of the group
  const bool lora = A != nullptr && i0 < rows;
  float* up = xs + static_cast<size_t>(rpc) * n;
  __nv_bfloat16* As = (lora && r2 * n * 2 <= kMaxAPrefetch)
                          ? reinterpret_cast<__nv_bfloat16*>(up + static_cast<size_t>(rpc) * r2)
                          : nullptr;
  if (As) prefetch_a_slice(A, d, c0, n, r2, As);
  pdl_wait();
  pdl_launch_dependents();
  for (int i = warp; i < rows; i += kRowWarps) {
    const size_t off = static_cast<size_t>(row0 + i) * d + c0;
    float* xr = xs + static_cast<size_t>(i) * n;
    float ss = 0.f;
    for (int e0 = 4 * lane; e0 < n; e0 += 128 * kRowUnroll) {
      // every load of the chunk is issued before the first use
      float4 v[kRowUnroll];
      uint2 q[kRowUnroll];
#pragma unroll
      for (int k = 0; k < kRowUnroll; ++k) {
        const int e = e0 + 128 * k;
        if (e < n) {
          v[k] = *reinterpret_cast<const float4*>(h + off + e);
          if (RESID) q[k] = *reinterpret_cast<const uint2*>(y + off + e);
        }
      }
#pragma unroll
      for (int k = 0; k < kRowUnroll; ++k) {
        const int e = e0 + 128 * k;
        if (e < n) {
          if (RESID) {
            const float2 y01 = unpack_bf16x2(q[k].x), y23 = unpack_bf16x2(q[k].y);
            v[k].x += y01.x;
            v[k].y += y01.y;
            v[k].z += y23.x;
            v[k].w += y23.y;
            *reinterpret_cast<float4*>(h + off + e) = v[k];
          }
          *reinterpret_cast<float4*>(xr + e) = v[k];
          ss += v[k].x * v[k].x + v[k].y * v[k].y + v[k].z * v[k].z + v[k].w * v[k].w;
        }
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if (lane == 0) ssq[i] = ss;
  }
  cluster_sync_all();
  for (int i = warp; i < rows; i += kRowWarps) {
    // the ranks' partial sums of squares, added in rank order
    const float mine = lane < kCl ? ld_cluster_f32(&ssq[i], static_cast<uint32_t>(lane)) : 0.f;
    float tot = 0.f;
    for (int q = 0; q < kCl; ++q) tot += __shfl_sync(0xffffffffu, mine, q);
    const float inv = rsqrtf(tot / static_cast<float>(d) + eps);
    const size_t off = static_cast<size_t>(row0 + i) * d + c0;
    float* xr = xs + static_cast<size_t>(i) * n;
    for (int e0 = 4 * lane; e0 < n; e0 += 128 * kRowUnroll) {
      uint2 wq[kRowUnroll];
#pragma unroll
      for (int k = 0; k < kRowUnroll; ++k)
        if (e0 + 128 * k < n) wq[k] = __ldg(reinterpret_cast<const uint2*>(w + c0 + e0 + 128 * k));
#pragma unroll
      for (int k = 0; k < kRowUnroll; ++k) {
        const int e = e0 + 128 * k;
        if (e >= n) continue;
        const float4 v = *reinterpret_cast<const float4*>(xr + e);
        const float2 w01 = unpack_bf16x2(wq[k].x), w23 = unpack_bf16x2(wq[k].y);
        const uint32_t o0 = pack_bf16x2(v.x * inv * w01.x, v.y * inv * w01.y);
        const uint32_t o1 = pack_bf16x2(v.z * inv * w23.x, v.w * inv * w23.y);
        *reinterpret_cast<uint2*>(a + off + e) = make_uint2(o0, o1);
        const float2 b01 = unpack_bf16x2(o0), b23 = unpack_bf16x2(o1);
        *reinterpret_cast<float4*>(xr + e) = make_float4(b01.x, b01.y, b23.x, b23.y);
      }
    }
  }
  if (As) wait_a_slice();
  else __syncthreads();
  if (lora)
    lora_group(xs, rows, i0, n, c0, d, A, As, r2, s, up, u, row0 + i0 - S, rank);
  else
    cluster_sync_all();  // the same cluster barriers on every path
  cluster_sync_all();    // remote reads of up finish before any CTA leaves
}

// The draw of one step (Algorithm 1: the actor samples each sequence's next token; the
// reference head's log-probability of it feeds the KL reward, and the critic head's value is
// kept with it). One thread-block cluster of kSampleCl CTAs per sequence s; CTA `rank` owns a
// 1/kSampleCl slice of the vocabulary and of the value head's d inputs. In one pass over its
// slice a thread keeps, for both heads, a running maximum and the sum of exp(z - max) (the
// sum rescaled when the maximum moves), and the first maximum of z + Gumbel noise. The
// per-thread, per-warp and per-CTA partials are merged in a fixed order (the CTAs' into rank
// 0 through distributed shared memory), so the result does not depend on timing; the argmax
// takes the lowest index among equal keys.
constexpr int kSampleCl = 8;
constexpr int kSampleThreads = 512;
constexpr int kSampleWarps = kSampleThreads / 32;
constexpr int kSampleBatch = 2;  // float4 loads per array and thread in flight together

struct SamplePart {
  float m_on, l_on, m_off, l_off, key, v;
  int idx;
};

__device__ __forceinline__ void lse_add(float& m, float& l, float z) {
  if (z > m) {
    l = l * expf(m - z) + 1.f;  // 0 * 0 + 1 on the first finite z
    m = z;
  } else if (z > -INFINITY) {
    l += expf(z - m);
  }
}
__device__ __forceinline__ void lse_merge(float& m, float& l, float m2, float l2) {
  const float M = fmaxf(m, m2);
  if (M == -INFINITY) return;  // both sides empty
  l = l * expf(m - M) + l2 * expf(m2 - M);
  m = M;
}
__device__ __forceinline__ void argmax_merge(float& key, int& idx, float k2, int i2) {
  if (k2 > key || (k2 == key && i2 < idx)) {
    key = k2;
    idx = i2;
  }
}
__device__ __forceinline__ void sample_merge(SamplePart& a, const SamplePart& b) {
  lse_merge(a.m_on, a.l_on, b.m_on, b.l_on);
  lse_merge(a.m_off, a.l_off, b.m_off, b.l_off);
  argmax_merge(a.key, a.idx, b.key, b.idx);
  a.v += b.v;
}
__device__ __forceinline__ SamplePart shfl_part(const SamplePart& p, int o) {
  SamplePart q;
  q.m_on = __shfl_xor_sync(0xffffffffu, p.m_on, o);
  q.l_on = __shfl_xor_sync(0xffffffffu, p.l_on, o);
  q.m_off = __shfl_xor_sync(0xffffffffu, p.m_off, o);
  q.l_off = __shfl_xor_sync(0xffffffffu, p.l_off, o);
  q.key = __shfl_xor_sync(0xffffffffu, p.key, o);
  q.v = __shfl_xor_sync(0xffffffffu, p.v, o);
  q.idx = __shfl_xor_sync(0xffffffffu, p.idx, o);
  return q;
}

// Cluster (kSampleCl, 1, 1) per sequence s: the drawn token of step t = *step from the
// actor's logits (row S + s) plus the step's Gumbel noise (none: greedy), its log-probability
// under both heads (the reference head is row s), and the value w_rm . fin[S + s].
// V % 4 == 0 (16-byte rows).
__global__ void __launch_bounds__(kSampleThreads)
    sample_tokens_kernel(const float* __restrict__ logits, int S, int V,
                         const float* __restrict__ gumbel, const __nv_bfloat16* __restrict__ fin,
                         int d, const __nv_bfloat16* __restrict__ w_rm,
                         const int* __restrict__ step, int n_steps, int32_t* __restrict__ tokens,
                         float* __restrict__ logp_a, float* __restrict__ logp_r,
                         float* __restrict__ values, int32_t* __restrict__ cur_ids) {
  __shared__ SamplePart warp_part[kSampleWarps];
  __shared__ float recv[kSampleCl][8];  // rank 0: every CTA's partial (idx as its bits)
  pdl_wait();
  pdl_launch_dependents();
  const int t = *step;
  if (t < 0 || t >= n_steps) return;  // grid-uniform; the host launches exactly n_steps draws
  cluster_arrive_relaxed();
  const uint32_t rank = cluster_rank();
  const int s = blockIdx.x / kSampleCl;
  const float* zo = logits + static_cast<size_t>(S + s) * V;
  const float* zr = logits + static_cast<size_t>(s) * V;
  const float* gn = gumbel ? gumbel + (static_cast<size_t>(t) * S + s) * V : nullptr;
  const int V4 = V / 4;
  const int chunk4 = (V4 + kSampleCl - 1) / kSampleCl;
  const int b4 = min(V4, static_cast<int>(rank) * chunk4), e4 = min(V4, b4 + chunk4);

  SamplePart p = {-INFINITY, 0.f, -INFINITY, 0.f, -INFINITY, 0.f, V};
  for (int q0 = b4 + threadIdx.x; q0 < e4; q0 += kSampleBatch * kSampleThreads) {
    float4 a[kSampleBatch], b[kSampleBatch], g[kSampleBatch];
#pragma unroll
    for (int j = 0; j < kSampleBatch; ++j) {
      const int q = q0 + j * kSampleThreads;
      if (q < e4) {
        a[j] = reinterpret_cast<const float4*>(zo)[q];
        b[j] = reinterpret_cast<const float4*>(zr)[q];
        g[j] = gn ? reinterpret_cast<const float4*>(gn)[q] : make_float4(0.f, 0.f, 0.f, 0.f);
      }
    }
#pragma unroll
    for (int j = 0; j < kSampleBatch; ++j) {
      const int q = q0 + j * kSampleThreads;
      if (q >= e4) break;
      const float av[4] = {a[j].x, a[j].y, a[j].z, a[j].w};
      const float bv[4] = {b[j].x, b[j].y, b[j].z, b[j].w};
      const float gv[4] = {g[j].x, g[j].y, g[j].z, g[j].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        lse_add(p.m_on, p.l_on, av[e]);
        lse_add(p.m_off, p.l_off, bv[e]);
        const float kk = gn ? av[e] + gv[e] : av[e];
        if (kk > p.key) {  // indices increase along a thread: the first maximum is kept
          p.key = kk;
          p.idx = 4 * q + e;
        }
      }
    }
  }
  // this CTA's slice of the value head
  const int dchunk = (d + kSampleCl - 1) / kSampleCl;
  const int d0 = min(d, static_cast<int>(rank) * dchunk), d1 = min(d, d0 + dchunk);
  const __nv_bfloat16* f = fin + static_cast<size_t>(S + s) * d;
  for (int k = d0 + threadIdx.x; k < d1; k += kSampleThreads)
    p.v = fmaf(__bfloat162float(f[k]), __bfloat162float(w_rm[k]), p.v);

#pragma unroll
  for (int o = 1; o < 32; o <<= 1) sample_merge(p, shfl_part(p, o));
  const int warp = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) warp_part[warp] = p;
  __syncthreads();
  cluster_wait();  // every CTA of the cluster has started: rank 0's shared memory is live
  if (threadIdx.x == 0) {
    SamplePart c = warp_part[0];
    for (int w = 1; w < kSampleWarps; ++w) sample_merge(c, warp_part[w]);
    const float vals[8] = {c.m_on, c.l_on, c.m_off, c.l_off, c.key, __int_as_float(c.idx), c.v, 0.f};
#pragma unroll
    for (int k = 0; k < 7; ++k) st_cluster_f32(&recv[rank][k], 0, vals[k]);
  }
  cluster_sync_all();
  if (rank != 0 || threadIdx.x != 0) return;
  SamplePart c = {recv[0][0], recv[0][1], recv[0][2], recv[0][3], recv[0][4], recv[0][6],
                  __float_as_int(recv[0][5])};
  for (int q = 1; q < kSampleCl; ++q) {
    const SamplePart o = {recv[q][0], recv[q][1], recv[q][2], recv[q][3], recv[q][4], recv[q][6],
                          __float_as_int(recv[q][5])};
    sample_merge(c, o);
  }
  const int tok = c.idx < V ? c.idx : 0;
  const size_t o = static_cast<size_t>(s) * n_steps + t;
  tokens[o] = tok;
  logp_a[o] = zo[tok] - (c.m_on + logf(c.l_on));
  logp_r[o] = zr[tok] - (c.m_off + logf(c.l_off));
  values[o] = c.v;
  cur_ids[s] = tok;
}



}  // namespace

int launch_kv_store_prefill(const void* qkv, int64_t R, int64_t P0, int64_t ld, int64_t d,
                            int64_t H, int64_t Pmax, void* ck, void* cv, cudaStream_t st) {
  if (R * P0 == 0) return 0;
  kv_store_prefill_kernel<<<static_cast<unsigned>(R * P0), 256, 0, st>>>(
      static_cast<const __nv_bfloat16*>(qkv), static_cast<int>(P0), static_cast<int>(ld),
      static_cast<int>(d), static_cast<int>(H), static_cast<int>(Pmax),
      static_cast<__nv_bfloat16*>(ck), static_cast<__nv_bfloat16*>(cv));
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

size_t decode_attention_smem(int64_t Pmax) {
  return static_cast<size_t>(Pmax) * 4 + static_cast<size_t>(kAttnWarps) * kDh * 4;
}

int launch_decode_attention(void* qkv, int64_t R, int64_t ld, int64_t d, int64_t H,
                            const void* table, void* ck, void* cv, int64_t P0, const int* step,
                            int64_t Pmax, void* out, int64_t ld_out, cudaStream_t st) {
  if (R == 0) return 0;
  const size_t smem = decode_attention_smem(Pmax);
  // up to 16 rows the single-pass kernel (4 sequences: decode step 3.685 -> 3.541 ms against
  // the two-pass kernel with pipelined key loads, which had taken it from 3.755 to 3.617);
  // above, the two-pass kernel with one iteration's loads at a time (pipelined loads were
  // slower at 12, 32 and 64 sequences: 4.38 against 4.18 ms, 5.62 against 5.58 ms,
  // 7.37-7.44 against 7.26 ms)
  if (R <= kGemvMaxRows) {
    const size_t smem1 = static_cast<size_t>(kAttnStages) * kAttnStageBytes;  // > the partials
    static bool attr1 = false;
    if (!attr1) {
      if (cudaFuncSetAttribute(decode_attention_1p_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               static_cast<int>(smem1)) != cudaSuccess)
        return -1;
      attr1 = true;
    }
    const cudaError_t e1 = launch_pdl(
        decode_attention_1p_kernel, dim3(static_cast<unsigned>(H), static_cast<unsigned>(R)),
        dim3(kAttnThreads), smem1, st, static_cast<const __nv_bfloat16*>(qkv), static_cast<int>(ld),
        static_cast<int>(d), static_cast<int>(H), static_cast<const float2*>(table),
        static_cast<__nv_bfloat16*>(ck), static_cast<__nv_bfloat16*>(cv), static_cast<int>(P0),
        step, static_cast<int>(Pmax),
        1.4426950408889634f / sqrtf(static_cast<float>(kDh)), static_cast<__nv_bfloat16*>(out),
        static_cast<int>(ld_out));
    return e1 == cudaSuccess ? 0 : -3;
  }
  auto kernel = decode_attention_kernel;
  static size_t attr = 0;
  if (smem > 48 * 1024 && smem > attr) {
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem)) != cudaSuccess)
      return -1;
    attr = smem;
  }
  const cudaError_t e = launch_pdl(
      kernel, dim3(static_cast<unsigned>(H), static_cast<unsigned>(R)),
      dim3(kAttnThreads), smem, st, static_cast<const __nv_bfloat16*>(qkv), static_cast<int>(ld),
      static_cast<int>(d), static_cast<int>(H), static_cast<const float2*>(table),
      static_cast<__nv_bfloat16*>(ck), static_cast<__nv_bfloat16*>(cv), static_cast<int>(P0),
      step, static_cast<int>(Pmax),
      1.0f / sqrtf(static_cast<float>(kDh)), static_cast<__nv_bfloat16*>(out),
      static_cast<int>(ld_out));
  return e == cudaSuccess ? 0 : -3;
}



// Raise a kernel's dynamic shared-memory limit when a launch needs more than the default
// (once per kernel and size: `done` remembers the largest limit set).
static int set_smem_limit(const void* kernel, size_t bytes, size_t& done) {
  if (bytes <= 48 * 1024 || bytes <= done) return 0;
  if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(bytes)) != cudaSuccess)
    return -1;
  done = bytes;
  return 0;
}

// cudaLaunchKernelEx with a (cl, 1, 1) cluster of `threads`-thread CTAs (by default the row
// kernels' kCl CTAs of kRowThreads) and programmatic dependent launch
template <typename... KArgs, typename... Args>
static cudaError_t launch_cluster_n(void (*kernel)(KArgs...), dim3 grid, unsigned threads,
                                    unsigned cl, size_t smem, cudaStream_t st, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(threads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cl;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}
template <typename... KArgs, typename... Args>
static cudaError_t launch_cluster(void (*kernel)(KArgs...), dim3 grid, size_t smem,
                                  cudaStream_t st, Args&&... args) {
  return launch_cluster_n(kernel, grid, kRowThreads, kCl, smem, st, std::forward<Args>(args)...);
}

int launch_sample_tokens(const float* logits, int64_t S, int64_t V, const float* gumbel,
                         const void* fin, int64_t d, const void* w_rm, const int* step,
                         int64_t n_steps, int32_t* tokens, float* logp_a, float* logp_r,
                         float* values, int32_t* cur_ids, cudaStream_t st) {
  if (S == 0) return 0;
  if (V % 4 != 0) return -1;
  const cudaError_t e = launch_cluster_n(
      sample_tokens_kernel, dim3(static_cast<unsigned>(S * kSampleCl)), kSampleThreads, kSampleCl,
      0, st, logits, static_cast<int>(S), static_cast<int>(V), gumbel,
      static_cast<const __nv_bfloat16*>(fin), static_cast<int>(d),
      static_cast<const __nv_bfloat16*>(w_rm), step, static_cast<int>(n_steps), tokens, logp_a,
      logp_r, values, cur_ids);
  return e == cudaSuccess ? 0 : -3;
}

int launch_row_norm_lora(float* h, const void* y, const void* w, int64_t R, int64_t d, float eps,
                         void* a, int64_t S, const void* A, int64_t r2, float s, void* u,
                         cudaStream_t st) {
  if (R == 0) return 0;
  if (d % (8 * kCl) != 0 || r2 > kMaxR2) return -1;
  const size_t n = static_cast<size_t>(d / kCl);
  const size_t a_bytes = n * 2 * static_cast<size_t>(r2);
  if (R >= kGroupMinRows) {
    const int rpc = static_cast<int>(std::min<int64_t>(kMaxRpc, (R + kGroupRowsPerCta - 1) / kGroupRowsPerCta));
    const size_t gsmem = static_cast<size_t>(rpc) * (n + static_cast<size_t>(r2)) * 4 +
                         (A != nullptr && a_bytes <= kMaxAPrefetch ? a_bytes : 0);
    static size_t gdone_resid = 0, gdone_plain = 0;
    if (set_smem_limit(y != nullptr ? reinterpret_cast<const void*>(row_norm_lora_group_kernel<true>)
                                    : reinterpret_cast<const void*>(row_norm_lora_group_kernel<false>),
                       gsmem, y != nullptr ? gdone_resid : gdone_plain) != 0)
      return -1;
    const dim3 grid(kCl, static_cast<unsigned>((R + rpc - 1) / rpc));
    const cudaError_t e =
        y != nullptr
            ? launch_cluster(row_norm_lora_group_kernel<true>, grid, gsmem, st, h,
                             static_cast<const __nv_bfloat16*>(y), static_cast<const __nv_bfloat16*>(w),
                             static_cast<int>(R), rpc, static_cast<int>(d), eps,
                             static_cast<__nv_bfloat16*>(a), static_cast<int>(S),
                             static_cast<const __nv_bfloat16*>(A), static_cast<int>(r2), s,
                             static_cast<__nv_bfloat16*>(u))
            : launch_cluster(row_norm_lora_group_kernel<false>, grid, gsmem, st, h,
                             static_cast<const __nv_bfloat16*>(nullptr),
                             static_cast<const __nv_bfloat16*>(w), static_cast<int>(R), rpc,
                             static_cast<int>(d), eps, static_cast<__nv_bfloat16*>(a),
                             static_cast<int>(S), static_cast<const __nv_bfloat16*>(A),
                             static_cast<int>(r2), s, static_cast<__nv_bfloat16*>(u));
    return e == cudaSuccess ? 0 : -3;
  }
  const size_t smem = n * 4 + (A != nullptr && a_bytes <= kMaxAPrefetch ? a_bytes : 0);
  static size_t done_resid = 0, done_plain = 0;
  if (set_smem_limit(y != nullptr ? reinterpret_cast<const void*>(row_norm_lora_kernel<true>)
                                  : reinterpret_cast<const void*>(row_norm_lora_kernel<false>),
                     smem, y != nullptr ? done_resid : done_plain) != 0)
    return -1;
  const dim3 grid(kCl, static_cast<unsigned>(R));
  cudaError_t e;
  if (y != nullptr)
    e = launch_cluster(row_norm_lora_kernel<true>, grid, smem, st, h,
                       static_cast<const __nv_bfloat16*>(y), static_cast<const __nv_bfloat16*>(w),
                       static_cast<int>(d), eps, static_cast<__nv_bfloat16*>(a), static_cast<int>(S),
                       static_cast<const __nv_bfloat16*>(A), static_cast<int>(r2), s,
                       static_cast<__nv_bfloat16*>(u));
  else
    e = launch_cluster(row_norm_lora_kernel<false>, grid, smem, st, h,
                       static_cast<const __nv_bfloat16*>(nullptr), static_cast<const __nv_bfloat16*>(w),
                       static_cast<int>(d), eps, static_cast<__nv_bfloat16*>(a), static_cast<int>(S),
                       static_cast<const __nv_bfloat16*>(A), static_cast<int>(r2), s,
                       static_cast<__nv_bfloat16*>(u));
  return e == cudaSuccess ? 0 : -3;
}

int launch_swiglu_lora(const void* gu, int64_t R, int64_t F, void* m, int64_t S, const void* A,
                       int64_t r, float s, void* u, cudaStream_t st) {
  if (R == 0) return 0;
  if (F % (8 * kCl) != 0 || r > kMaxR2) return -1;
  const size_t n = static_cast<size_t>(F / kCl);
  const size_t a_bytes = n * 2 * static_cast<size_t>(r);
  const size_t smem = n * 4 + (A != nullptr && a_bytes <= kMaxAPrefetch ? a_bytes : 0);
  static size_t done = 0;
  if (set_smem_limit(reinterpret_cast<const void*>(swiglu_lora_kernel), smem, done) != 0) return -1;
  const cudaError_t e = launch_cluster(
      swiglu_lora_kernel, dim3(kCl, static_cast<unsigned>(R)), smem, st,
      static_cast<const __nv_bfloat16*>(gu), static_cast<int>(F), static_cast<__nv_bfloat16*>(m),
      static_cast<int>(S), static_cast<const __nv_bfloat16*>(A), static_cast<int>(r), s,
      static_cast<__nv_bfloat16*>(u));
  return e == cudaSuccess ? 0 : -3;
}


}  // namespace hydra
