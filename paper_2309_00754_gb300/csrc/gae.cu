// Reverse GAE scan, one warp per sequence (§2: GAE builds the advantage estimates from
// V(x, y); the critic is trained on the returns. Appendix B: gamma = 1.0, lambda = 0.95).
//
//   delta_t = r_t + gamma V_{t+1} [t + 1 < len] - V_t
//   A_t     = delta_t + gamma lambda A_{t+1},   A_len = 0
//   R_t     = A_t + V_t;   A_t = R_t = 0 for t >= len
//
// General lengths: the warp loads its sequence into shared memory with coalesced loads.
// Lane j owns the contiguous chunk [j c, j c + c). Each lane runs the recursion over its chunk with a zero
// carry, which gives an affine map A_start = b + m A_next (m = (gamma lambda)^count). A
// warp-shuffle suffix scan composes the 32 maps, every lane then adds its carry-in times
// the matching power of gamma lambda, and the results leave through coalesced stores.
#include "common.cuh"
#include "kernels.h"

namespace hydra {
namespace {

__global__ void gae_scan_kernel(const float* __restrict__ rew, const float* __restrict__ val,
                                const int32_t* __restrict__ lengths, int S, int L, int chunk,
                                int stride, int warps_per_block, float gamma, float lam,
                                float* __restrict__ adv, float* __restrict__ ret, int* err) {
  extern __shared__ float sm[];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int s = blockIdx.x * warps_per_block + warp;
  if (s >= S) return;
  float* rb = sm + static_cast<size_t>(warp) * 2 * 32 * stride;
  float* vb = rb + 32 * stride;

  int n = lengths ? lengths[s] : L;
  if (n < 0 || n > L) {
    if (lane == 0) record_error(err, kDevBadLength);
    n = n < 0 ? 0 : L;
  }
  const float* rr = rew + static_cast<size_t>(s) * L;
  const float* vv = val + static_cast<size_t>(s) * L;
  for (int t = lane; t < n; t += 32) {
    const int j = t / chunk;
    const int o = j * stride + (t - j * chunk);
    rb[o] = __ldcs(rr + t);
    vb[o] = __ldcs(vv + t);
  }
  __syncwarp();

  const float c = gamma * lam;
  const int lo = lane * chunk;
  const int he = min(min(L, lo + chunk), n);  // end of this lane's valid range
  float* rl = rb + lane * stride;
  float* vl = vb + lane * stride;

  // value following the chunk: first element of the next chunk when it is still valid
  float v_next = (he < n) ? vb[(lane + 1) * stride] : 0.f;
  float a = 0.f;
  float m = 1.f;
  for (int t = he - 1; t >= lo; --t) {
    const float vt = vl[t - lo];
    const float delta = rl[t - lo] + gamma * v_next - vt;
    a = delta + c * a;
    rl[t - lo] = a;  // local advantage with a zero carry
    m *= c;
    v_next = vt;
  }
  float b = (he > lo) ? a : 0.f;

  // inclusive suffix scan of the maps X_j = b_j + m_j X_{j+1}
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float b2 = __shfl_down_sync(0xffffffffu, b, off);
    const float m2 = __shfl_down_sync(0xffffffffu, m, off);
    if (lane + off < 32) {
      b = fmaf(m, b2, b);
      m *= m2;
    }
  }
  float carry = __shfl_down_sync(0xffffffffu, b, 1);
  if (lane == 31) carry = 0.f;

  float p = c;
  for (int t = he - 1; t >= lo; --t) {
    const float at = fmaf(p, carry, rl[t - lo]);
    rl[t - lo] = at;
    vl[t - lo] = at + vl[t - lo];
    p *= c;
  }
  __syncwarp();

  float* ao = adv + static_cast<size_t>(s) * L;
  float* ro = ret + static_cast<size_t>(s) * L;
  for (int t = lane; t < L; t += 32) {
    float av = 0.f, rv = 0.f;
    if (t < n) {
      const int j = t / chunk;
      const int o = j * stride + (t - j * chunk);
      av = rb[o];
      rv = vb[o];
    }
    __stcs(ao + t, av);
    __stcs(ro + t, rv);
  }
}

// Register-only variant for L = 32 CH (CH % 4 == 0, L <= 512): lane l owns elements
// [CH l, CH l + CH), loaded and stored as float4 (rows are 16-byte aligned); the value after
// the chunk comes from lane l + 1 by shuffle. float4 groups at or beyond the sequence length
// are neither read nor computed.
template <int CH>
__global__ void __launch_bounds__(256)
    gae_scan_reg_kernel(const float* __restrict__ rew, const float* __restrict__ val,
                        const int32_t* __restrict__ lengths, int S, float gamma, float lam,
                        float* __restrict__ adv, float* __restrict__ ret, int* err) {
  constexpr int L = 32 * CH;
  const int lane = threadIdx.x & 31;
  const int s = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (s >= S) return;
  int n = lengths ? lengths[s] : L;
  if (n < 0 || n > L) {
    if (lane == 0) record_error(err, kDevBadLength);
    n = n < 0 ? 0 : L;
  }
  const int lo = lane * CH;
  const float4* rr = reinterpret_cast<const float4*>(rew + static_cast<size_t>(s) * L + lo);
  const float4* vv = reinterpret_cast<const float4*>(val + static_cast<size_t>(s) * L + lo);
  float r[CH], v[CH];
#pragma unroll
  for (int q = 0; q < CH / 4; ++q) {
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f), b = a;
    if (lo + 4 * q < n) {
      a = __ldcs(rr + q);
      b = __ldcs(vv + q);
    }
    r[4 * q] = a.x; r[4 * q + 1] = a.y; r[4 * q + 2] = a.z; r[4 * q + 3] = a.w;
    v[4 * q] = b.x; v[4 * q + 1] = b.y; v[4 * q + 2] = b.z; v[4 * q + 3] = b.w;
  }
  const float c = gamma * lam;
  // value following this lane's chunk: the next lane's first value while still valid
  const float v_after = __shfl_down_sync(0xffffffffu, v[0], 1);
  const int he = min(lo + CH, n);
  float a = 0.f, m = 1.f;
  float loc[CH];
#pragma unroll
  for (int i = CH - 1; i >= 0; --i) {
    const int t = lo + i;
    loc[i] = 0.f;
    if (t < he) {
      const float vn = (i == CH - 1) ? ((t + 1 < n) ? v_after : 0.f) : ((t + 1 < n) ? v[i + 1] : 0.f);
      a = (r[i] + gamma * vn - v[i]) + c * a;
      loc[i] = a;
      m *= c;
    }
  }
  float b = (he > lo) ? a : 0.f;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float b2 = __shfl_down_sync(0xffffffffu, b, off);
    const float m2 = __shfl_down_sync(0xffffffffu, m, off);
    if (lane + off < 32) {
      b = fmaf(m, b2, b);
      m *= m2;
    }
  }
  float carry = __shfl_down_sync(0xffffffffu, b, 1);
  if (lane == 31) carry = 0.f;
  float p = c;
#pragma unroll
  for (int i = CH - 1; i >= 0; --i) {
    if (lo + i < he) {
      loc[i] = fmaf(p, carry, loc[i]);
      p *= c;
    }
  }
  float4* ao = reinterpret_cast<float4*>(adv + static_cast<size_t>(s) * L + lo);
  float4* ro = reinterpret_cast<float4*>(ret + static_cast<size_t>(s) * L + lo);
#pragma unroll
  for (int q = 0; q < CH / 4; ++q) {
    float e[4], f[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const bool ok = lo + 4 * q + k < n;
      e[k] = ok ? loc[4 * q + k] : 0.f;
      f[k] = ok ? loc[4 * q + k] + v[4 * q + k] : 0.f;
    }
    __stcs(ao + q, make_float4(e[0], e[1], e[2], e[3]));
    __stcs(ro + q, make_float4(f[0], f[1], f[2], f[3]));
  }
}

}  // namespace

int launch_gae(const float* r, const float* v, const int32_t* lengths, int64_t S, int64_t L,
               float gamma, float lam, float* adv, float* ret, int* err, cudaStream_t stream) {
  if (S == 0 || L == 0) return 0;
  const bool aligned = (reinterpret_cast<uintptr_t>(r) % 16 == 0) &&
                       (reinterpret_cast<uintptr_t>(v) % 16 == 0) &&
                       (reinterpret_cast<uintptr_t>(adv) % 16 == 0) &&
                       (reinterpret_cast<uintptr_t>(ret) % 16 == 0);
  if (aligned && L % 128 == 0 && L <= 512) {
    const unsigned grid = static_cast<unsigned>((S + 7) / 8);
    const int si = static_cast<int>(S);
    switch (L / 32) {
      case 4: gae_scan_reg_kernel<4><<<grid, 256, 0, stream>>>(r, v, lengths, si, gamma, lam, adv, ret, err); break;
      case 8: gae_scan_reg_kernel<8><<<grid, 256, 0, stream>>>(r, v, lengths, si, gamma, lam, adv, ret, err); break;
      case 12: gae_scan_reg_kernel<12><<<grid, 256, 0, stream>>>(r, v, lengths, si, gamma, lam, adv, ret, err); break;
      default: gae_scan_reg_kernel<16><<<grid, 256, 0, stream>>>(r, v, lengths, si, gamma, lam, adv, ret, err); break;
    }
    return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
  }
  const int chunk = static_cast<int>((L + 31) / 32);
  const int stride = (chunk & 1) ? chunk : chunk + 1;  // odd stride: conflict-free lanes
  const size_t per_warp = static_cast<size_t>(2) * 32 * stride * sizeof(float);
  int wpb = static_cast<int>((96 * 1024) / per_warp);
  wpb = wpb < 1 ? 1 : (wpb > 8 ? 8 : wpb);
  const size_t smem = per_warp * wpb;
  static size_t attr_bytes = 0;
  if (smem > 48 * 1024 && smem > attr_bytes) {
    if (cudaFuncSetAttribute(gae_scan_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem)) != cudaSuccess)
      return -1;
    attr_bytes = smem;
  }
  const unsigned grid = static_cast<unsigned>((S + wpb - 1) / wpb);
  gae_scan_kernel<<<grid, 32 * wpb, smem, stream>>>(r, v, lengths, static_cast<int>(S),
                                                   static_cast<int>(L), chunk, stride, wpb, gamma,
                                                   lam, adv, ret, err);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace hydra
