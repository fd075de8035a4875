// Kernels of the KV-cached generation loop (Algorithms 1 and 2: "generate sequence using the
// policy for T steps"; J-Hydra-PPO keeps the critic head's value of every step). The decode
// step runs the R = 2 S stacked rows of the LoRA-off and LoRA-on streams of S sequences; the
// projections are the dual-output GEMV, the rest is here:
//   kv_store_prefill   the prompt's rotated keys and its values into the cache
//   decode_rope_append rotary embedding of the new token's q and k, k and v appended
//   decode_attention   one query row per (row, head) against the cached positions 0..pos
//   swiglu_blocked     SwiGLU on gate/up columns interleaved in blocks of 128
//   sample_tokens      per sequence: log-softmax of both heads, the Gumbel-max draw from the
//                      actor's logits, both log-probabilities of the drawn token, the value
// The step counter lives in device memory, so one captured step replays for every position.
// Cache layout per layer: K [R][H][Pmax][Dh] then V [R][H][Pmax][Dh], bf16, row i = stream
// * S + sequence.
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

// One block per stacked row: q rotated in place, k rotated into the cache, v copied. The same
// explicit roundings as the prefill's rotary (no contraction), from the same table.
__global__ void decode_rope_append_kernel(__nv_bfloat16* __restrict__ qkv, int ld, int d, int H,
                                          const float2* __restrict__ table, int P0,
                                          const int* __restrict__ step, int Pmax,
                                          __nv_bfloat16* __restrict__ ck,
                                          __nv_bfloat16* __restrict__ cv) {
  const int i = blockIdx.x;
  const int pos = P0 + *step - 1;
  if (pos < 0 || pos >= Pmax) return;  // the host keeps every step inside the cache
  __nv_bfloat16* row = qkv + static_cast<size_t>(i) * ld;
  const float2* tb = table + static_cast<size_t>(pos) * (kDh / 2);
  constexpr int half = kDh / 2;
  for (int e = threadIdx.x; e < 2 * H * half; e += blockDim.x) {
    const int blk = e / (H * half);  // 0: q, 1: k
    const int r = e - blk * H * half;
    const int h = r / half, j = r % half;
    __nv_bfloat16* x = row + blk * d + h * kDh;
    const float x1 = __bfloat162float(x[j]), x2 = __bfloat162float(x[j + half]);
    const float c = tb[j].x, s = tb[j].y;
    const __nv_bfloat16 o1 = __float2bfloat16_rn(__fsub_rn(__fmul_rn(x1, c), __fmul_rn(x2, s)));
    const __nv_bfloat16 o2 = __float2bfloat16_rn(__fadd_rn(__fmul_rn(x1, s), __fmul_rn(x2, c)));
    if (blk == 0) {
      x[j] = o1;
      x[j + half] = o2;
    } else {
      __nv_bfloat16* dst = ck + ((static_cast<size_t>(i) * H + h) * Pmax + pos) * kDh;
      dst[j] = o1;
      dst[j + half] = o2;
    }
  }
  for (int e = threadIdx.x * 8; e < d; e += blockDim.x * 8) {
    const int h = e / kDh, j = e % kDh;
    *reinterpret_cast<uint4*>(cv + ((static_cast<size_t>(i) * H + h) * Pmax + pos) * kDh + j) =
        *reinterpret_cast<const uint4*>(row + 2 * d + e);
  }
}

constexpr int kAttnThreads = 128;
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

// One block per (head, row): scores of the npos = pos + 1 cached keys into shared memory
// (groups of 8 lanes per key, 32 bytes each, reduced by shuffles), the softmax over them,
// then the weighted sum of the values (lane = 4 output dimensions, warps split positions).
__global__ void __launch_bounds__(kAttnThreads)
    decode_attention_kernel(const __nv_bfloat16* __restrict__ qkv, int ld, int H,
                            const __nv_bfloat16* __restrict__ ck,
                            const __nv_bfloat16* __restrict__ cv, int P0,
                            const int* __restrict__ step, int Pmax, float scale,
                            __nv_bfloat16* __restrict__ out, int ld_out) {
  extern __shared__ float sc[];  // [Pmax] scores, then [kAttnWarps][kDh] partial outputs
  __shared__ float red[kAttnWarps];
  const int h = blockIdx.x, i = blockIdx.y;
  const int npos = min(P0 + *step, Pmax);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const __nv_bfloat16* K = ck + (static_cast<size_t>(i) * H + h) * Pmax * kDh;
  const __nv_bfloat16* Vc = cv + (static_cast<size_t>(i) * H + h) * Pmax * kDh;
  const int g = lane >> 3, sub = lane & 7;
  float qf[16];
  {
    const __nv_bfloat16* q = qkv + static_cast<size_t>(i) * ld + h * kDh + 16 * sub;
    const uint4 a = *reinterpret_cast<const uint4*>(q);
    const uint4 b = *reinterpret_cast<const uint4*>(q + 8);
    const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float2 f = unpack_bf16x2(w[k]);
      qf[2 * k] = f.x * scale;
      qf[2 * k + 1] = f.y * scale;
    }
  }
  // warp-uniform trip count: all 32 lanes reach the shuffles
  for (int base = warp * 4; base < npos; base += 4 * kAttnWarps) {
    const int p = base + g;
    uint4 a = make_uint4(0u, 0u, 0u, 0u), b = a;
    if (p < npos) {
      const __nv_bfloat16* kr = K + static_cast<size_t>(p) * kDh + 16 * sub;
      a = __ldcs(reinterpret_cast<const uint4*>(kr));
      b = __ldcs(reinterpret_cast<const uint4*>(kr + 8));
    }
    const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
    float acc = 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float2 f = unpack_bf16x2(w[k]);
      acc = fmaf(qf[2 * k], f.x, acc);
      acc = fmaf(qf[2 * k + 1], f.y, acc);
    }
    acc += __shfl_xor_sync(0xffffffffu, acc, 1);
    acc += __shfl_xor_sync(0xffffffffu, acc, 2);
    acc += __shfl_xor_sync(0xffffffffu, acc, 4);
    if (sub == 0 && p < npos) sc[p] = acc;
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
#pragma unroll 4
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

// gu [R, 2F]: column block 2b holds gate features 128b..128b+127, block 2b+1 the matching up
// features; m [R, F] = bf16(silu(gate) * up)
__global__ void swiglu_blocked_kernel(const __nv_bfloat16* __restrict__ gu, long long R, int F,
                                      __nv_bfloat16* __restrict__ m) {
  const long long n8 = R * (F / 8);
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < n8;
       e += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long row = e / (F / 8);
    const int c = static_cast<int>(e - row * (F / 8)) * 8;  // output feature
    const int b = c / 128, j = c % 128;
    const __nv_bfloat16* base = gu + static_cast<size_t>(row) * 2 * F + 256 * b + j;
    const uint4 g = *reinterpret_cast<const uint4*>(base);
    const uint4 u = *reinterpret_cast<const uint4*>(base + 128);
    const uint32_t* gp = &g.x;
    const uint32_t* up = &u.x;
    uint4 o;
    uint32_t* op = &o.x;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float2 gf = unpack_bf16x2(gp[k]);
      const float2 uf = unpack_bf16x2(up[k]);
      op[k] = pack_bf16x2(gf.x / (1.0f + expf(-gf.x)) * uf.x, gf.y / (1.0f + expf(-gf.y)) * uf.y);
    }
    *reinterpret_cast<uint4*>(m + static_cast<size_t>(row) * F + c) = o;
  }
}

constexpr int kSampleThreads = 512;

// Block s: the drawn token of sequence s at step t = *step from the actor's logits (row
// S + s) plus the step's Gumbel noise (none: greedy), its log-probability under both heads
// (the reference head is row s), and the value w_rm . fin[S + s].
__global__ void __launch_bounds__(kSampleThreads)
    sample_tokens_kernel(const float* __restrict__ logits, int S, int V,
                         const float* __restrict__ gumbel, const __nv_bfloat16* __restrict__ fin,
                         int d, const __nv_bfloat16* __restrict__ w_rm,
                         const int* __restrict__ step, int n_steps, int32_t* __restrict__ tokens,
                         float* __restrict__ logp_a, float* __restrict__ logp_r,
                         float* __restrict__ values, int32_t* __restrict__ cur_ids) {
  __shared__ float red[kSampleThreads / 32];
  __shared__ float bkey[kSampleThreads / 32];
  __shared__ int bidx[kSampleThreads / 32];
  const int s = blockIdx.x;
  const int t = *step;
  if (t < 0 || t >= n_steps) return;  // the host launches exactly n_steps draws
  const float* zo = logits + static_cast<size_t>(S + s) * V;
  const float* zr = logits + static_cast<size_t>(s) * V;
  const float* gn = gumbel ? gumbel + (static_cast<size_t>(t) * S + s) * V : nullptr;
  float m_on = -INFINITY, m_off = -INFINITY, key = -INFINITY;
  int idx = V;
  for (int k = threadIdx.x; k < V; k += kSampleThreads) {
    const float a = zo[k], b = zr[k];
    m_on = fmaxf(m_on, a);
    m_off = fmaxf(m_off, b);
    const float kk = gn ? a + gn[k] : a;
    if (kk > key) {  // k increases: the first maximum of this thread's stripe
      key = kk;
      idx = k;
    }
  }
  // argmax across the block, ties to the lowest index
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float k2 = __shfl_xor_sync(0xffffffffu, key, o);
    const int i2 = __shfl_xor_sync(0xffffffffu, idx, o);
    if (k2 > key || (k2 == key && i2 < idx)) {
      key = k2;
      idx = i2;
    }
  }
  const int warp = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) {
    bkey[warp] = key;
    bidx[warp] = idx;
  }
  m_on = block_max(m_on, red);
  m_off = block_max(m_off, red);
  key = bkey[0];
  idx = bidx[0];
  for (int w = 1; w < kSampleThreads / 32; ++w)
    if (bkey[w] > key || (bkey[w] == key && bidx[w] < idx)) {
      key = bkey[w];
      idx = bidx[w];
    }
  float l_on = 0.f, l_off = 0.f;
  for (int k = threadIdx.x; k < V; k += kSampleThreads) {
    l_on += expf(zo[k] - m_on);
    l_off += expf(zr[k] - m_off);
  }
  l_on = block_sum(l_on, red);
  l_off = block_sum(l_off, red);
  const __nv_bfloat16* f = fin + static_cast<size_t>(S + s) * d;
  float v = 0.f;
  for (int k = threadIdx.x; k < d; k += kSampleThreads)
    v = fmaf(__bfloat162float(f[k]), __bfloat162float(w_rm[k]), v);
  v = block_sum(v, red);
  if (threadIdx.x == 0) {
    const int tok = idx < V ? idx : 0;
    const size_t o = static_cast<size_t>(s) * n_steps + t;
    tokens[o] = tok;
    logp_a[o] = zo[tok] - (m_on + logf(l_on));
    logp_r[o] = zr[tok] - (m_off + logf(l_off));
    values[o] = v;
    cur_ids[s] = tok;
  }
}

__global__ void step_advance_kernel(int* step) { *step += 1; }

int grid_for(long long n, int block) {
  long long g = (n + block - 1) / block;
  if (g > 65535LL * 8) g = 65535LL * 8;
  return static_cast<int>(g < 1 ? 1 : g);
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

int launch_decode_rope_append(void* qkv, int64_t R, int64_t ld, int64_t d, int64_t H,
                              const void* table, int64_t P0, const int* step, int64_t Pmax,
                              void* ck, void* cv, cudaStream_t st) {
  if (R == 0) return 0;
  decode_rope_append_kernel<<<static_cast<unsigned>(R), 256, 0, st>>>(
      static_cast<__nv_bfloat16*>(qkv), static_cast<int>(ld), static_cast<int>(d),
      static_cast<int>(H), static_cast<const float2*>(table), static_cast<int>(P0), step,
      static_cast<int>(Pmax), static_cast<__nv_bfloat16*>(ck), static_cast<__nv_bfloat16*>(cv));
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

size_t decode_attention_smem(int64_t Pmax) {
  return static_cast<size_t>(Pmax) * 4 + static_cast<size_t>(kAttnWarps) * kDh * 4;
}

int launch_decode_attention(const void* qkv, int64_t R, int64_t ld, int64_t H, const void* ck,
                            const void* cv, int64_t P0, const int* step, int64_t Pmax, void* out,
                            int64_t ld_out, cudaStream_t st) {
  if (R == 0) return 0;
  const size_t smem = decode_attention_smem(Pmax);
  static size_t attr = 0;
  if (smem > 48 * 1024 && smem > attr) {
    if (cudaFuncSetAttribute(decode_attention_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem)) != cudaSuccess)
      return -1;
    attr = smem;
  }
  decode_attention_kernel<<<dim3(static_cast<unsigned>(H), static_cast<unsigned>(R)), kAttnThreads,
                            smem, st>>>(
      static_cast<const __nv_bfloat16*>(qkv), static_cast<int>(ld), static_cast<int>(H),
      static_cast<const __nv_bfloat16*>(ck), static_cast<const __nv_bfloat16*>(cv),
      static_cast<int>(P0), step, static_cast<int>(Pmax), 1.0f / sqrtf(static_cast<float>(kDh)),
      static_cast<__nv_bfloat16*>(out), static_cast<int>(ld_out));
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

int launch_swiglu_blocked(const void* gu, int64_t R, int64_t F, void* m, cudaStream_t st) {
  if (R == 0) return 0;
  swiglu_blocked_kernel<<<grid_for(R * (F / 8), 256), 256, 0, st>>>(
      static_cast<const __nv_bfloat16*>(gu), R, static_cast<int>(F), static_cast<__nv_bfloat16*>(m));
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

int launch_sample_tokens(const float* logits, int64_t S, int64_t V, const float* gumbel,
                         const void* fin, int64_t d, const void* w_rm, const int* step,
                         int64_t n_steps, int32_t* tokens, float* logp_a, float* logp_r,
                         float* values, int32_t* cur_ids, cudaStream_t st) {
  if (S == 0) return 0;
  sample_tokens_kernel<<<static_cast<unsigned>(S), kSampleThreads, 0, st>>>(
      logits, static_cast<int>(S), static_cast<int>(V), gumbel,
      static_cast<const __nv_bfloat16*>(fin), static_cast<int>(d),
      static_cast<const __nv_bfloat16*>(w_rm), step, static_cast<int>(n_steps), tokens, logp_a,
      logp_r, values, cur_ids);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

int launch_step_advance(int* step, cudaStream_t st) {
  step_advance_kernel<<<1, 1, 0, st>>>(step);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace hydra
