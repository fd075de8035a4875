// Memory-bound pieces of the Llama decoder used by the full Hydra scoring pass (the paper
// runs Llama 7b, §4): token embedding, RMSNorm, rotary embedding, SwiGLU, residual add and
// the scalar reward/value head. The residual stream is fp32; every tensor that feeds a
// matrix product is bf16. Rows of the two streams (LoRA off / LoRA on) are stacked, so
// each kernel covers both streams in one launch.
#include <float.h>

#include "common.cuh"
#include "kernels.h"

namespace hydra {
namespace {

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

// row i of the output reads row (i / g_out) * g_in + off + i % g_out of the input
__device__ __forceinline__ long long map_row(long long i, const RowMap& m) {
  return (i / m.g_out) * m.g_in + m.off + (i % m.g_out);
}

// ---------------------------------------------------------------- embedding

// h[s T + t] = fp32(table[ids[t]]) for s < copies; a NaN row and an error code for an id
// outside the vocabulary. With `step` (the decode loop's device-side step counter), block 0
// also advances the counter: the token just drawn moves to the next position.
__global__ void embed_kernel(const __nv_bfloat16* __restrict__ table, int V, int d,
                             const int32_t* __restrict__ ids, long long T, int copies,
                             float* __restrict__ h, int* err, int* step) {
  pdl_wait();
  pdl_launch_dependents();
  const long long t = blockIdx.x;
  if (step != nullptr && t == 0 && threadIdx.x == 0) *step += 1;
  const int id = ids[t];
  const bool bad = id < 0 || id >= V;
  if (bad && threadIdx.x == 0) record_error(err, kDevBadTokenId);
  const uint4* src = reinterpret_cast<const uint4*>(table + static_cast<size_t>(bad ? 0 : id) * d);
  for (int c = threadIdx.x; c < d / 8; c += blockDim.x) {
    float f[8];
    const uint4 v = __ldg(src + c);
    float2 a = unpack_bf16x2(v.x), b = unpack_bf16x2(v.y), e = unpack_bf16x2(v.z),
           g = unpack_bf16x2(v.w);
    f[0] = a.x; f[1] = a.y; f[2] = b.x; f[3] = b.y; f[4] = e.x; f[5] = e.y; f[6] = g.x; f[7] = g.y;
    if (bad) {
#pragma unroll
      for (int j = 0; j < 8; ++j) f[j] = __int_as_float(0x7fc00000);
    }
    for (int s = 0; s < copies; ++s) {
      float4* dst = reinterpret_cast<float4*>(h + (static_cast<size_t>(s) * T + t) * d) + 2 * c;
      dst[0] = make_float4(f[0], f[1], f[2], f[3]);
      dst[1] = make_float4(f[4], f[5], f[6], f[7]);
    }
  }
}

// ---------------------------------------------------------------- RMSNorm

// y[i] = bf16( x[map(i)] / sqrt(mean(x^2) + eps) * w ), one CTA of 128 threads per row
__global__ void __launch_bounds__(128)
    rmsnorm_kernel(const float* __restrict__ x, const __nv_bfloat16* __restrict__ w, int d,
                   float eps, RowMap map, __nv_bfloat16* __restrict__ y) {
  const long long i = blockIdx.x;
  const float4* xr = reinterpret_cast<const float4*>(x + static_cast<size_t>(map_row(i, map)) * d);
  const int n4 = d / 4;
  float ss = 0.f;
  for (int c = threadIdx.x; c < n4; c += 128) {
    const float4 v = xr[c];
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  ss = warp_sum(ss);
  __shared__ float red[4];
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  const float tot = red[0] + red[1] + red[2] + red[3];
  const float inv = rsqrtf(tot / static_cast<float>(d) + eps);
  uint2* yr = reinterpret_cast<uint2*>(y + static_cast<size_t>(i) * d);
  const uint2* wr = reinterpret_cast<const uint2*>(w);
  for (int c = threadIdx.x; c < n4; c += 128) {
    const float4 v = xr[c];
    const uint2 wv = __ldg(wr + c);
    const float2 w01 = unpack_bf16x2(wv.x), w23 = unpack_bf16x2(wv.y);
    uint2 o;
    o.x = pack_bf16x2(v.x * inv * w01.x, v.y * inv * w01.y);
    o.y = pack_bf16x2(v.z * inv * w23.x, v.w * inv * w23.y);
    yr[c] = o;
  }
}

// ---------------------------------------------------------------- rotary embedding

// In place on the q and k blocks of each row of qkv ([R, ld] bf16; q at column 0, k at
// column d). Rotate-half pairing: dims (i, i + Dh/2) of each head rotate by
// pos * theta^(-2i/Dh), pos = row % P (position within its sequence). One warp per row;
// lane l owns the pair indices i = 2l, 2l + 1 (+ 64 l' for Dh > 128), computes their angles
// once and applies them to every head of q and k with 4-byte (bf16 x 2) accesses.
__global__ void __launch_bounds__(128)
    rope_kernel(__nv_bfloat16* __restrict__ qkv, long long R, int ld, int d, int Dh, int P,
                float log2_theta) {
  const long long row = blockIdx.x * 4LL + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= R) return;
  const int half = Dh / 2;
  const float pos = static_cast<float>(row % P);
  __nv_bfloat16* base = qkv + static_cast<size_t>(row) * ld;
  const int heads = d / Dh;
  for (int i = 2 * lane; i < half; i += 64) {
    float c0, s0, c1, s1;
    sincosf(pos * exp2f(-(2.0f * i / Dh) * log2_theta), &s0, &c0);
    sincosf(pos * exp2f(-(2.0f * (i + 1) / Dh) * log2_theta), &s1, &c1);
    for (int hb = 0; hb < 2 * heads; ++hb) {  // q heads then k heads (k block starts at d)
      uint32_t* p1 = reinterpret_cast<uint32_t*>(base + hb * Dh + i);
      uint32_t* p2 = reinterpret_cast<uint32_t*>(base + hb * Dh + i + half);
      const float2 x1 = unpack_bf16x2(*p1), x2 = unpack_bf16x2(*p2);
      // explicit roundings (no contraction), so the rotary epilogue of the tcgen05 GEMM, which
      // runs the same operations, gives the same bits
      *p1 = pack_bf16x2(__fsub_rn(__fmul_rn(x1.x, c0), __fmul_rn(x2.x, s0)),
                        __fsub_rn(__fmul_rn(x1.y, c1), __fmul_rn(x2.y, s1)));
      *p2 = pack_bf16x2(__fadd_rn(__fmul_rn(x1.x, s0), __fmul_rn(x2.x, c0)),
                        __fadd_rn(__fmul_rn(x1.y, s1), __fmul_rn(x2.y, c1)));
    }
  }
}

// (cos a, sin a) for a = pos * theta^(-2i/Dh), pos in [0, P), pair i in [0, Dh/2): the rotation
// table of the fused rotary GEMM epilogue, the same expression as rope_kernel evaluates
__global__ void rope_table_kernel(long long n, int half, int Dh, float log2_theta,
                                  float2* __restrict__ table) {
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < n;
       e += static_cast<long long>(gridDim.x) * blockDim.x) {
    const float pos = static_cast<float>(e / half);
    const int i = static_cast<int>(e % half);
    float c, s;
    sincosf(pos * exp2f(-(2.0f * i / Dh) * log2_theta), &s, &c);
    table[e] = make_float2(c, s);
  }
}

// ---------------------------------------------------------------- SwiGLU

// gu: [R, 2F] bf16 (gate in [0, F), up in [F, 2F)); m = bf16(silu(gate) * up), [R, F]
__global__ void swiglu_kernel(const __nv_bfloat16* __restrict__ gu, long long R, int F,
                              __nv_bfloat16* __restrict__ m) {
  const long long n8 = R * (F / 8);
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < n8;
       e += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long row = e / (F / 8);
    const int c = static_cast<int>(e - row * (F / 8));
    const uint4 g = __ldg(reinterpret_cast<const uint4*>(gu + static_cast<size_t>(row) * 2 * F) + c);
    const uint4 u = __ldg(reinterpret_cast<const uint4*>(gu + static_cast<size_t>(row) * 2 * F + F) + c);
    const uint32_t* gp = &g.x;
    const uint32_t* up = &u.x;
    uint4 o;
    uint32_t* op = &o.x;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 gf = unpack_bf16x2(gp[j]);
      const float2 uf = unpack_bf16x2(up[j]);
      const float a = gf.x / (1.0f + expf(-gf.x)) * uf.x;
      const float b = gf.y / (1.0f + expf(-gf.y)) * uf.y;
      op[j] = pack_bf16x2(a, b);
    }
    reinterpret_cast<uint4*>(m + static_cast<size_t>(row) * F)[c] = o;
  }
}

// ---------------------------------------------------------------- residual add

// h[i] += float(y[i]) over n elements (n % 8 == 0)
__global__ void residual_add_kernel(float* __restrict__ h, const __nv_bfloat16* __restrict__ y,
                                    long long n) {
  const long long n8 = n / 8;
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < n8;
       e += static_cast<long long>(gridDim.x) * blockDim.x) {
    const uint4 v = __ldg(reinterpret_cast<const uint4*>(y) + e);
    float4* hp = reinterpret_cast<float4*>(h) + 2 * e;
    float4 a = hp[0], b = hp[1];
    const float2 p = unpack_bf16x2(v.x), q = unpack_bf16x2(v.y), r = unpack_bf16x2(v.z),
                 s = unpack_bf16x2(v.w);
    a.x += p.x; a.y += p.y; a.z += q.x; a.w += q.y;
    b.x += r.x; b.y += r.y; b.z += s.x; b.w += s.y;
    hp[0] = a;
    hp[1] = b;
  }
}

// ---------------------------------------------------------------- scalar head

// out[i] = sum_k x[map(i), k] w[k], one warp per output row (reward model / value head).
// With `lengths`, rows are [S, L] (i = s L + t) and rows t >= lengths[s] are written 0.
__global__ void head_dot_kernel(const __nv_bfloat16* __restrict__ x, int d,
                                const __nv_bfloat16* __restrict__ w, RowMap map, long long n,
                                const int32_t* __restrict__ lengths, int L,
                                float* __restrict__ out) {
  const long long i = blockIdx.x * 8LL + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (i >= n) return;
  if (lengths != nullptr && (i % L) >= lengths[i / L]) {
    if (lane == 0) out[i] = 0.f;
    return;
  }
  const uint4* xr = reinterpret_cast<const uint4*>(x + static_cast<size_t>(map_row(i, map)) * d);
  const uint4* wr = reinterpret_cast<const uint4*>(w);
  float acc = 0.f;
  for (int c = lane; c < d / 8; c += 32) {
    const uint4 a = __ldg(xr + c), b = __ldg(wr + c);
    const uint32_t* ap = &a.x;
    const uint32_t* bp = &b.x;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 fa = unpack_bf16x2(ap[j]), fb = unpack_bf16x2(bp[j]);
      acc = fmaf(fa.x, fb.x, acc);
      acc = fmaf(fa.y, fb.y, acc);
    }
  }
  acc = warp_sum(acc);
  if (lane == 0) out[i] = acc;
}

// ---------------------------------------------------------------- sequence score

// score[s] = w . bf16(RMSNorm(h[s P + p0 + len_s - 1]) * g): the reward-model head on the
// normed hidden state of the sequence's last valid token (0 when len_s == 0). One CTA of
// 128 threads per sequence.
__global__ void __launch_bounds__(128)
    seq_score_kernel(const float* __restrict__ h, const __nv_bfloat16* __restrict__ g,
                     const __nv_bfloat16* __restrict__ w, int d, float eps,
                     const int32_t* __restrict__ lengths, int L, long long P, long long p0,
                     float* __restrict__ score) {
  const int s = blockIdx.x;
  int n = lengths ? lengths[s] : L;
  n = n < 0 ? 0 : (n > L ? L : n);
  __shared__ float red[4];
  if (n == 0) {
    if (threadIdx.x == 0) score[s] = 0.f;
    return;
  }
  const float* x = h + (static_cast<size_t>(s) * P + p0 + n - 1) * d;
  float ss = 0.f;
  for (int k = threadIdx.x; k < d; k += 128) ss += x[k] * x[k];
  ss = warp_sum(ss);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  const float inv = rsqrtf((red[0] + red[1] + red[2] + red[3]) / static_cast<float>(d) + eps);
  __syncthreads();
  float acc = 0.f;
  for (int k = threadIdx.x; k < d; k += 128) {
    const float y = __bfloat162float(__float2bfloat16_rn(x[k] * inv * __bfloat162float(g[k])));
    acc = fmaf(y, __bfloat162float(w[k]), acc);
  }
  acc = warp_sum(acc);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) score[s] = red[0] + red[1] + red[2] + red[3];
}

// dst row i = src row map(i), one CTA per row, 16-byte pieces
__global__ void __launch_bounds__(128)
    gather_rows_kernel(const uint4* __restrict__ src, int chunks, RowMap map,
                       uint4* __restrict__ dst) {
  const long long i = blockIdx.x;
  const uint4* s = src + static_cast<size_t>(map_row(i, map)) * chunks;
  uint4* o = dst + static_cast<size_t>(i) * chunks;
  for (int c = threadIdx.x; c < chunks; c += 128) o[c] = s[c];
}

unsigned grid_for(long long work, int threads) {
  long long b = (work + threads - 1) / threads;
  if (b > 152LL * 16) b = 152LL * 16;
  return static_cast<unsigned>(b < 1 ? 1 : b);
}

}  // namespace

int launch_embed(const void* table, int64_t V, int64_t d, const int32_t* ids, int64_t T,
                 int copies, float* h, int* err, cudaStream_t st, int* step) {
  if (T == 0) return 0;
  if (step == nullptr) {
    embed_kernel<<<static_cast<unsigned>(T), 128, 0, st>>>(
        static_cast<const __nv_bfloat16*>(table), static_cast<int>(V), static_cast<int>(d), ids,
        T, copies, h, err, nullptr);
    return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
  }
  const cudaError_t e = launch_pdl(embed_kernel, dim3(static_cast<unsigned>(T)), dim3(128), 0, st,
                                   static_cast<const __nv_bfloat16*>(table), static_cast<int>(V),
                                   static_cast<int>(d), ids, static_cast<long long>(T), copies, h,
                                   err, step);
  return e == cudaSuccess ? 0 : -3;
}

int launch_rmsnorm(const float* x, const void* w, int64_t rows, int64_t d, float eps,
                   const RowMap& map, void* y, cudaStream_t st) {
  if (rows == 0) return 0;
  rmsnorm_kernel<<<static_cast<unsigned>(rows), 128, 0, st>>>(
      x, static_cast<const __nv_bfloat16*>(w), static_cast<int>(d), eps, map,
      static_cast<__nv_bfloat16*>(y));
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

int launch_rope(void* qkv, int64_t R, int64_t ld, int64_t d, int64_t Dh, int64_t P, float theta,
                cudaStream_t st) {
  if (R == 0) return 0;
  rope_kernel<<<static_cast<unsigned>((R + 3) / 4), 128, 0, st>>>(static_cast<__nv_bfloat16*>(qkv), R,
                                                        static_cast<int>(ld), static_cast<int>(d),
                                                        static_cast<int>(Dh), static_cast<int>(P),
                                                        log2f(theta));
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

int launch_rope_table(int64_t P, int64_t Dh, float theta, void* table, cudaStream_t st) {
  if (P == 0) return 0;
  const long long n = P * (Dh / 2);
  rope_table_kernel<<<grid_for(n, 256), 256, 0, st>>>(n, static_cast<int>(Dh / 2),
                                                      static_cast<int>(Dh), log2f(theta),
                                                      static_cast<float2*>(table));
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

int launch_swiglu(const void* gu, int64_t R, int64_t F, void* m, cudaStream_t st) {
  if (R == 0) return 0;
  swiglu_kernel<<<grid_for(R * (F / 8), 256), 256, 0, st>>>(
      static_cast<const __nv_bfloat16*>(gu), R, static_cast<int>(F), static_cast<__nv_bfloat16*>(m));
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

int launch_residual_add(float* h, const void* y, int64_t n, cudaStream_t st) {
  if (n == 0) return 0;
  residual_add_kernel<<<grid_for(n / 8, 256), 256, 0, st>>>(h, static_cast<const __nv_bfloat16*>(y), n);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

int launch_head_dot(const void* x, int64_t d, const void* w, const RowMap& map, int64_t n,
                    const int32_t* lengths, int64_t L, float* out, cudaStream_t st) {
  if (n == 0) return 0;
  head_dot_kernel<<<static_cast<unsigned>((n + 7) / 8), 256, 0, st>>>(
      static_cast<const __nv_bfloat16*>(x), static_cast<int>(d),
      static_cast<const __nv_bfloat16*>(w), map, n, lengths, static_cast<int>(L), out);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

int launch_gather_rows(const void* src, int64_t rows, int64_t row_bytes, const RowMap& map,
                       void* dst, cudaStream_t st) {
  if (rows == 0) return 0;
  if (row_bytes % 16 != 0) return -4;
  gather_rows_kernel<<<static_cast<unsigned>(rows), 128, 0, st>>>(
      static_cast<const uint4*>(src), static_cast<int>(row_bytes / 16), map,
      static_cast<uint4*>(dst));
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

int launch_seq_score(const float* h, const void* norm, const void* w, int64_t d, float eps,
                     const int32_t* lengths, int64_t S, int64_t L, int64_t P, int64_t p0,
                     float* score, cudaStream_t st) {
  if (S == 0) return 0;
  seq_score_kernel<<<static_cast<unsigned>(S), 128, 0, st>>>(
      h, static_cast<const __nv_bfloat16*>(norm), static_cast<const __nv_bfloat16*>(w),
      static_cast<int>(d), eps, lengths, static_cast<int>(L), P, p0, score);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace hydra
