// Update side of PPO over the scored batch (§2 "Stage 3: PPO"; Algorithms 1 and 2 optimise
// the surrogate after scoring). Per valid token t < len_s of an [S, L] batch:
//
//   r_t   = exp(logp_new_t - logp_old_t)                   probability ratio r(theta)
//   A_t   = adv_t, or (adv_t - mean) / sqrt(M2 / n + 1e-8)   with advantage whitening
//   s_t   = min(r_t A_t, clip(r_t, 1 - eps, 1 + eps) A_t)   clipped surrogate term
//   loss_clip  = -(1/n) sum s_t,   d/d logp_new_t = -r_t A_t / n where r_t A_t <= clip term
//   loss_value =  (1/n) sum (V_t - R_t)^2,   d/d V_t = 2 (V_t - R_t) / n
//
// Up to four launches, chained with programmatic dependent launch:
//   moments:  per block, the valid count n and (with whitening) the sums of a - c and
//             (a - c)^2 over the valid advantages, c = adv[0] a common shift;
//   coef:     one block merges those partials (or takes the caller's moments) into
//             (mean, 1 / std, 1 / n);
//   loss:     streams float4 chunks of the flattened [S, L] batch, several chunks' loads
//             in flight per thread; chunks past a row's length are written as zero
//             gradients without reading the inputs; per-block sums go to the workspace;
//   finalize: one block merges the per-block sums, in a fixed order, and writes the
//             statistics.
// Every grid is one wave (SMs x resident blocks), so no block waits for a second wave.
// Per-thread sums are compensated (Kahan) fp32, block and cross-block trees fp32: GB300
// executes fp64 at a small fraction of its fp32 rate, so fp64 appears only in a few scalar
// operations of the output.
// HBM-bound: the loss pass reads 20 B per valid token and writes 8 B per token of the
// [S, L] gradient arrays; the moments pass reads 4 B per valid token with whitening.
#include "common.cuh"
#include "kernels.h"

namespace hydra {
namespace {

constexpr int kPpoThreads = 256;
constexpr int kPpoWarps = kPpoThreads / 32;
constexpr int kLossSums = 5;  // sum s, sum (V-R)^2, sum kl, sum a, sum a^2 (+ clipped count)

// Workspace layout: moments partials, loss partials, then the merged moments.
struct MomPart {
  int n;
  float s1, s2, pad;  // sums of (a - c) and (a - c)^2
};
struct LossPart {
  int nclip;
  float s[kLossSums];
  float pad[2];
};

// Partials written by the previous launch are read through L2 (ld.global.cg).
__device__ __forceinline__ MomPart load_part(const MomPart* p) {
  const int4 q = __ldcg(reinterpret_cast<const int4*>(p));
  return MomPart{q.x, __int_as_float(q.y), __int_as_float(q.z), 0.f};
}
__device__ __forceinline__ LossPart load_part(const LossPart* p) {
  const int4 a = __ldcg(reinterpret_cast<const int4*>(p));
  const int4 b = __ldcg(reinterpret_cast<const int4*>(p) + 1);
  return LossPart{a.x, {__int_as_float(a.y), __int_as_float(a.z), __int_as_float(a.w),
                        __int_as_float(b.x), __int_as_float(b.y)}, {0.f, 0.f}};
}

struct Kahan {
  float s = 0.f, c = 0.f;
  __device__ __forceinline__ void add(float x) {
    const float y = x - c;
    const float t = s + y;
    c = (t - s) - y;
    s = t;
  }
};

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ int warp_sum_i(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Fixed-shape block sums of N floats and one int; results valid in every thread.
template <int N>
__device__ __forceinline__ void block_sums(float (&v)[N], int& k, float (*sh)[kPpoWarps],
                                           int* shk) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int i = 0; i < N; ++i) v[i] = warp_sum(v[i]);
  k = warp_sum_i(k);
  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < N; ++i) sh[i][warp] = v[i];
    shk[warp] = k;
  }
  __syncthreads();
#pragma unroll
  for (int i = 0; i < N; ++i) {
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < kPpoWarps; ++w) t += sh[i][w];
    v[i] = t;
  }
  int t = 0;
#pragma unroll
  for (int w = 0; w < kPpoWarps; ++w) t += shk[w];
  k = t;
  __syncthreads();
}

__device__ __forceinline__ int clamp_length(int n, int L, int* err) {
  if (n < 0 || n > L) {
    record_error(err, kDevBadLength);
    n = n < 0 ? 0 : L;
  }
  return n;
}

__device__ __forceinline__ int row_length(const int32_t* lengths, int s, int L, int* err) {
  return clamp_length(lengths ? __ldg(lengths + s) : L, L, err);
}

// A thread's position in the flattened batch: row s, chunk column t (chunk q = s C + t),
// and row s's length, fetched one batch ahead so that its latency overlaps the previous
// batch's data loads. Advancing by a fixed number of chunks steps rows and columns without
// a division.
struct Cursor {
  int s, t, len;
};

__device__ __forceinline__ int fetch_length(const int32_t* lengths, int s, int S, int L) {
  return s < S ? (lengths ? __ldg(lengths + s) : L) : 0;
}

__device__ __forceinline__ Cursor cursor_at(unsigned q, int C, const int32_t* lengths, int S,
                                            int L) {
  const int s = static_cast<int>(q / static_cast<unsigned>(C));
  return Cursor{s, static_cast<int>(q - static_cast<unsigned>(s) * C), fetch_length(lengths, s, S, L)};
}

__device__ __forceinline__ void cursor_advance(Cursor& c, int ds, int dt, int C,
                                               const int32_t* lengths, int S, int L) {
  c.t += dt;
  c.s += ds;
  if (c.t >= C) {
    c.t -= C;
    ++c.s;
  }
  c.len = fetch_length(lengths, c.s, S, L);
}

template <int VEC>
struct Vec;
template <>
struct Vec<4> {
  static __device__ __forceinline__ void get(const float* p, float* v) {
    const float4 q = __ldcs(reinterpret_cast<const float4*>(p));
    v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
  }
  static __device__ __forceinline__ void put(float* p, const float* v) {
    __stcs(reinterpret_cast<float4*>(p), make_float4(v[0], v[1], v[2], v[3]));
  }
};
template <>
struct Vec<1> {
  static __device__ __forceinline__ void get(const float* p, float* v) { v[0] = __ldcs(p); }
  static __device__ __forceinline__ void put(float* p, const float* v) { __stcs(p, v[0]); }
};

// Loads that keep their lines in L2 (normal eviction priority): the moments pass reads the
// advantages this way, so that the loss pass, which reads them again with the rest of its
// inputs streaming (evict-first), finds them there when the batch fits in L2.
template <int VEC>
__device__ __forceinline__ void get_keep(const float* p, float* v) {
  if constexpr (VEC == 4) {
    const float4 q = __ldg(reinterpret_cast<const float4*>(p));
    v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
  } else {
    v[0] = __ldg(p);
  }
}

// Pass 1: valid count and shifted advantage sums per block. Chunk q of the flattened batch
// covers tokens [VEC (q mod C), +VEC) of row q / C, C = L / VEC. Each thread holds two
// batches of kMomBatch chunks: the next batch's loads are issued before the current one is
// added, so that two batches per thread are in flight.
constexpr int kMomBatch = 4;

template <int VEC>
struct MomBatch {
  float v[kMomBatch][VEC];
  int k[kMomBatch];  // valid tokens of each chunk
};

template <int VEC>
__device__ __forceinline__ void mom_load(MomBatch<VEC>& x, Cursor (&cur)[kMomBatch],
                                         const float* adv, int S, int L, int C, int ds, int dt,
                                         const int32_t* lengths, int* err) {
#pragma unroll
  for (int b = 0; b < kMomBatch; ++b) {
    x.k[b] = 0;
    if (cur[b].s < S) {
      const int t0 = cur[b].t * VEC;
      const int len = clamp_length(cur[b].len, L, t0 == 0 ? err : nullptr);
      x.k[b] = min(max(len - t0, 0), VEC);
      if (x.k[b] > 0) get_keep<VEC>(adv + static_cast<size_t>(cur[b].s) * L + t0, x.v[b]);
    }
  }
#pragma unroll
  for (int b = 0; b < kMomBatch; ++b) cursor_advance(cur[b], ds, dt, C, lengths, S, L);
}

template <int VEC>
__device__ __forceinline__ void mom_add(const MomBatch<VEC>& x, float c, int& n, Kahan& s1,
                                        Kahan& s2) {
  float b1 = 0.f, b2 = 0.f;  // this batch's sums, then one compensated add each
#pragma unroll
  for (int b = 0; b < kMomBatch; ++b)
#pragma unroll
    for (int j = 0; j < VEC; ++j) {
      const float d = j < x.k[b] ? x.v[b][j] - c : 0.f;
      b1 += d;
      b2 += d * d;
    }
#pragma unroll
  for (int b = 0; b < kMomBatch; ++b) n += x.k[b];
  s1.add(b1);
  s2.add(b2);
}

template <int VEC>
__global__ void __launch_bounds__(kPpoThreads, 3)
    ppo_moments_kernel(const float* __restrict__ adv, const int32_t* __restrict__ lengths, int S,
                       int L, int with_adv, MomPart* __restrict__ part, int* err) {
  __shared__ float sh[2][kPpoWarps];
  __shared__ int shk[kPpoWarps];
  pdl_wait();
  const unsigned tid = blockIdx.x * kPpoThreads + threadIdx.x;
  const unsigned nthr = gridDim.x * kPpoThreads;
  int n = 0;
  Kahan s1, s2;
  if (!with_adv) {
    for (unsigned s = tid; s < static_cast<unsigned>(S); s += nthr)
      n += row_length(lengths, static_cast<int>(s), L, err);
  } else if (L >= VEC) {  // C = L / VEC >= 1: the cursors divide by C
    const float c = S > 0 ? __ldg(adv) : 0.f;
    const int C = L / VEC;
    const unsigned step = kMomBatch * nthr;  // chunks per batch over the grid
    const int ds = static_cast<int>(step / C), dt = static_cast<int>(step % C);
    Cursor cur[kMomBatch];
#pragma unroll
    for (int b = 0; b < kMomBatch; ++b) cur[b] = cursor_at(tid + b * nthr, C, lengths, S, L);
    MomBatch<VEC> x, y;
    mom_load(x, cur, adv, S, L, C, ds, dt, lengths, err);
    while (true) {
      if (cur[0].s >= S) {
        mom_add(x, c, n, s1, s2);
        break;
      }
      mom_load(y, cur, adv, S, L, C, ds, dt, lengths, err);
      mom_add(x, c, n, s1, s2);
      if (cur[0].s >= S) {
        mom_add(y, c, n, s1, s2);
        break;
      }
      mom_load(x, cur, adv, S, L, C, ds, dt, lengths, err);
      mom_add(y, c, n, s1, s2);
    }
  }
  float v[2] = {s1.s, s2.s};
  block_sums<2>(v, n, sh, shk);
  if (threadIdx.x == 0) part[blockIdx.x] = MomPart{n, v[0], v[1], 0.f};
  pdl_launch_dependents();
}

// Pass 1, float4 rows (L % 4 == 0, aligned): one warp per row, two rows in flight per warp;
// lane l loads tokens [4 l + 128 k, + 4) of a row's valid prefix, k < 4 at a time, and the
// next pair's lengths are fetched before the current pair is added. A row's tokens past its
// length are never read.
__global__ void __launch_bounds__(kPpoThreads)
    ppo_moments_rows_kernel(const float* __restrict__ adv, const int32_t* __restrict__ lengths,
                            int S, int L, MomPart* __restrict__ part, int* err) {
  __shared__ float sh[2][kPpoWarps];
  __shared__ int shk[kPpoWarps];
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int gw = blockIdx.x * kPpoWarps + (threadIdx.x >> 5);
  const int nw = gridDim.x * kPpoWarps;
  const float c = S > 0 ? __ldg(adv) : 0.f;
  int n = 0;
  Kahan s1, s2;
  auto len_of = [&](int s) { return s < S ? (lengths ? __ldg(lengths + s) : L) : 0; };
  int nlA = len_of(gw), nlB = len_of(gw + nw);
  for (int s0 = gw; s0 < S; s0 += 2 * nw) {
    const int sA = s0, sB = s0 + nw;
    const int lenA = clamp_length(nlA, L, lane == 0 ? err : nullptr);
    const int lenB = sB < S ? clamp_length(nlB, L, lane == 0 ? err : nullptr) : 0;
    nlA = len_of(s0 + 2 * nw);
    nlB = len_of(s0 + 3 * nw);
    const float* ra = adv + static_cast<size_t>(sA) * L;
    const float* rb = adv + static_cast<size_t>(sB < S ? sB : sA) * L;
    const int lmax = max(lenA, lenB);
    for (int base = 0; base < lmax; base += 512) {
      float va[4][4], vb[4][4];
      int ka[4], kb[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int t0 = base + 128 * k + 4 * lane;
        ka[k] = min(max(lenA - t0, 0), 4);
        kb[k] = min(max(lenB - t0, 0), 4);
        if (ka[k] > 0) get_keep<4>(ra + t0, va[k]);
        if (kb[k] > 0) get_keep<4>(rb + t0, vb[k]);
      }
      float b1 = 0.f, b2 = 0.f;
#pragma unroll
      for (int k = 0; k < 4; ++k)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float da = j < ka[k] ? va[k][j] - c : 0.f;
          const float db = j < kb[k] ? vb[k][j] - c : 0.f;
          b1 += da + db;
          b2 += da * da + db * db;
        }
#pragma unroll
      for (int k = 0; k < 4; ++k) n += ka[k] + kb[k];
      s1.add(b1);
      s2.add(b2);
    }
  }
  float v[2] = {s1.s, s2.s};
  block_sums<2>(v, n, sh, shk);
  if (threadIdx.x == 0) part[blockIdx.x] = MomPart{n, v[0], v[1], 0.f};
  pdl_launch_dependents();
}

// Merge the moments partials (or take the caller's fp64 [n, mean, M2]) into the fp64
// moments and the fp32 coefficients (mean, 1 / sqrt(var + 1e-8), 1 / n) of the loss pass.
// Every thread loads its few partials at once (compensated fp32), then a fixed block tree.
constexpr int kMaxPartsPerThread = (kPpoMaxLossBlocks + kPpoThreads - 1) / kPpoThreads;

__global__ void __launch_bounds__(kPpoThreads)
    ppo_coef_kernel(const float* __restrict__ adv, int S, int L, int shifted,
                    const MomPart* __restrict__ part, int G, const double* __restrict__ ext,
                    double* __restrict__ moments, float* __restrict__ coef) {
  __shared__ float sh[2][kPpoWarps];
  __shared__ int shk[kPpoWarps];
  pdl_wait();
  if (ext != nullptr) {
    if (threadIdx.x == 0) {
      const double n = __ldcg(ext), mean = __ldcg(ext + 1), m2 = __ldcg(ext + 2);
      moments[0] = n;
      moments[1] = mean;
      moments[2] = m2;
      const double var = n > 0.0 ? m2 / n : 0.0;
      coef[0] = static_cast<float>(mean);
      coef[1] = static_cast<float>(1.0 / sqrt(var + 1e-8));
      coef[2] = n > 0.0 ? static_cast<float>(1.0 / n) : 0.f;
    }
  } else {
    MomPart p[kMaxPartsPerThread];
#pragma unroll
    for (int i = 0; i < kMaxPartsPerThread; ++i) {
      const int j = threadIdx.x + i * kPpoThreads;
      p[i] = j < G ? load_part(part + j) : MomPart{0, 0.f, 0.f, 0.f};
    }
    int n = 0;
    Kahan k1, k2;
#pragma unroll
    for (int i = 0; i < kMaxPartsPerThread; ++i) {
      n += p[i].n;
      k1.add(p[i].s1);
      k2.add(p[i].s2);
    }
    float v[2] = {k1.s, k2.s};
    block_sums<2>(v, n, sh, shk);
    if (threadIdx.x == 0) {
      float mean = 0.f, m2 = 0.f;
      if (n > 0) {
        const float c = shifted && S > 0 && L > 0 ? __ldg(adv) : 0.f;
        const float d1 = v[0] / static_cast<float>(n);
        mean = c + d1;
        m2 = fmaxf(v[1] - d1 * v[0], 0.f);
      }
      const float var = n > 0 ? m2 / static_cast<float>(n) : 0.f;
      moments[0] = static_cast<double>(n);
      moments[1] = static_cast<double>(mean);
      moments[2] = static_cast<double>(m2);
      coef[0] = mean;
      coef[1] = rsqrtf(var + 1e-8f);
      coef[2] = n > 0 ? 1.f / static_cast<float>(n) : 0.f;
    }
  }
  pdl_launch_dependents();
}

// Pass 2: per-token terms and gradients. Each thread holds two chunks: the next chunk's
// five loads are issued before the current chunk is computed and stored.
template <int VEC>
struct LossChunk {
  float ln[VEC], lo[VEC], a[VEC], R[VEC], V[VEC];
  int k;         // valid tokens; -1: past the end of the batch
  unsigned off;  // element offset (S * L < 2^31)
};

struct LossAcc {
  Kahan s, v, kl, a, aa;
  int nclip = 0;
};

template <int VEC>
__device__ __forceinline__ void loss_load(LossChunk<VEC>& x, Cursor& cur, const float* logp_new,
                                          const float* logp_old, const float* adv,
                                          const float* ret, const float* val, int S, int L,
                                          int C, int ds, int dt, const int32_t* lengths,
                                          int* err) {
  x.k = -1;
  x.off = 0;
  if (cur.s < S) {
    const int t0 = cur.t * VEC;
    const int len = clamp_length(cur.len, L, t0 == 0 ? err : nullptr);
    x.k = min(max(len - t0, 0), VEC);
    x.off = static_cast<unsigned>(cur.s) * static_cast<unsigned>(L) + t0;
    if (x.k > 0) {
      Vec<VEC>::get(logp_new + x.off, x.ln);
      Vec<VEC>::get(logp_old + x.off, x.lo);
      Vec<VEC>::get(adv + x.off, x.a);
      Vec<VEC>::get(ret + x.off, x.R);
      Vec<VEC>::get(val + x.off, x.V);
    }
  }
  cursor_advance(cur, ds, dt, C, lengths, S, L);
}

template <int VEC, bool WHITEN>
__device__ __forceinline__ void loss_compute(const LossChunk<VEC>& x, float mean, float inv_std,
                                             float inv_n, float eps, LossAcc& acc,
                                             float* grad_logp, float* grad_val) {
  if (x.k < 0) return;
  const float lo_clip = 1.f - eps, hi_clip = 1.f + eps;
  float gl[VEC], gv[VEC];
  float bs = 0.f, bv = 0.f, bkl = 0.f, ba = 0.f, baa = 0.f;  // this chunk's sums
#pragma unroll
  for (int j = 0; j < VEC; ++j) {
    gl[j] = gv[j] = 0.f;
    if (j < x.k) {
      const float d = x.ln[j] - x.lo[j];
      const float r = expf(d);
      const float A = WHITEN ? (x.a[j] - mean) * inv_std : x.a[j];
      const float rc = fminf(fmaxf(r, lo_clip), hi_clip);
      const float u = r * A, c = rc * A;
      const float dv = x.V[j] - x.R[j];
      bs += fminf(u, c);
      bv += dv * dv;
      bkl -= d;
      ba += x.a[j];
      baa += x.a[j] * x.a[j];
      acc.nclip += fabsf(r - 1.f) > eps ? 1 : 0;
      gl[j] = u <= c ? -u * inv_n : 0.f;
      gv[j] = 2.f * dv * inv_n;
    }
  }
  Vec<VEC>::put(grad_logp + x.off, gl);
  Vec<VEC>::put(grad_val + x.off, gv);
  if (x.k > 0) {
    acc.s.add(bs);
    acc.v.add(bv);
    acc.kl.add(bkl);
    acc.a.add(ba);
    acc.aa.add(baa);
  }
}

template <int VEC, bool WHITEN>
__global__ void __launch_bounds__(kPpoThreads, 3)
    ppo_loss_kernel(const float* __restrict__ logp_new, const float* __restrict__ logp_old,
                    const float* __restrict__ adv, const float* __restrict__ ret,
                    const float* __restrict__ val, const int32_t* __restrict__ lengths, int S,
                    int L, float eps, const float* __restrict__ coef,
                    LossPart* __restrict__ lpart, float* __restrict__ grad_logp,
                    float* __restrict__ grad_val, int* err) {
  __shared__ float sh[kLossSums][kPpoWarps];
  __shared__ int shk[kPpoWarps];
  pdl_wait();
  const float mean = __ldcg(coef), inv_std = __ldcg(coef + 1), inv_n = __ldcg(coef + 2);
  const unsigned tid = blockIdx.x * kPpoThreads + threadIdx.x;
  const unsigned nthr = gridDim.x * kPpoThreads;
  // C >= 1 here: the host launches this pass only for S * L > 0 with L % VEC == 0
  const int C = L / VEC;
  const int ds = static_cast<int>(nthr / C), dt = static_cast<int>(nthr % C);
  Cursor cur = cursor_at(tid, C, lengths, S, L);
  LossAcc acc;
  LossChunk<VEC> x, y;
  loss_load(x, cur, logp_new, logp_old, adv, ret, val, S, L, C, ds, dt, lengths, err);
  while (true) {
    if (cur.s >= S) {
      loss_compute<VEC, WHITEN>(x, mean, inv_std, inv_n, eps, acc, grad_logp, grad_val);
      break;
    }
    loss_load(y, cur, logp_new, logp_old, adv, ret, val, S, L, C, ds, dt, lengths, err);
    loss_compute<VEC, WHITEN>(x, mean, inv_std, inv_n, eps, acc, grad_logp, grad_val);
    if (cur.s >= S) {
      loss_compute<VEC, WHITEN>(y, mean, inv_std, inv_n, eps, acc, grad_logp, grad_val);
      break;
    }
    loss_load(x, cur, logp_new, logp_old, adv, ret, val, S, L, C, ds, dt, lengths, err);
    loss_compute<VEC, WHITEN>(y, mean, inv_std, inv_n, eps, acc, grad_logp, grad_val);
  }
  float v[kLossSums] = {acc.s.s, acc.v.s, acc.kl.s, acc.a.s, acc.aa.s};
  int nclip = acc.nclip;
  block_sums<kLossSums>(v, nclip, sh, shk);
  if (threadIdx.x == 0) {
    LossPart p;
    p.nclip = nclip;
#pragma unroll
    for (int i = 0; i < kLossSums; ++i) p.s[i] = v[i];
    p.pad[0] = p.pad[1] = 0.f;
    lpart[blockIdx.x] = p;
  }
  pdl_launch_dependents();
}

// Pass 3: merge the G loss partials (every thread loads its few at once, compensated fp32,
// then a fixed block tree) and write the statistics.
__global__ void __launch_bounds__(kPpoThreads)
    ppo_finalize_kernel(const LossPart* __restrict__ lpart, int G, const double* __restrict__ mom,
                        int report_moments, double* __restrict__ stats) {
  __shared__ float sh[kLossSums][kPpoWarps];
  __shared__ int shk[kPpoWarps];
  pdl_wait();
  LossPart p[kMaxPartsPerThread];
#pragma unroll
  for (int i = 0; i < kMaxPartsPerThread; ++i) {
    const int j = threadIdx.x + i * kPpoThreads;
    if (j < G) {
      p[i] = load_part(lpart + j);
    } else {
      p[i] = LossPart{0, {0.f, 0.f, 0.f, 0.f, 0.f}, {0.f, 0.f}};
    }
  }
  int nclip = 0;
  Kahan acc[kLossSums];
#pragma unroll
  for (int i = 0; i < kMaxPartsPerThread; ++i) {
    nclip += p[i].nclip;
#pragma unroll
    for (int k = 0; k < kLossSums; ++k) acc[k].add(p[i].s[k]);
  }
  float v[kLossSums];
#pragma unroll
  for (int k = 0; k < kLossSums; ++k) v[k] = acc[k].s;
  block_sums<kLossSums>(v, nclip, sh, shk);
  if (threadIdx.x == 0) {
    const double n = __ldcg(mom), inv = n > 0.0 ? 1.0 / n : 0.0;
    stats[0] = -static_cast<double>(v[0]) * inv;
    stats[1] = static_cast<double>(v[1]) * inv;
    stats[2] = static_cast<double>(nclip) * inv;
    stats[3] = static_cast<double>(v[2]) * inv;
    if (report_moments) {
      stats[4] = __ldcg(mom + 1);
      stats[5] = n > 0.0 ? sqrt(__ldcg(mom + 2) * inv) : 0.0;
    } else {
      const double m = static_cast<double>(v[3]) * inv;
      stats[4] = m;
      stats[5] = n > 0.0 ? sqrt(fmax(static_cast<double>(v[4]) * inv - m * m, 0.0)) : 0.0;
    }
    stats[6] = n;
  }
}

int num_sms() {
  static int nsm = 0;
  if (nsm == 0) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      nsm = 148;
  }
  return nsm;
}

// One wave: SMs x resident blocks per SM (capped by the work and the workspace slots).
template <typename K>
int one_wave(K kernel, long long work_items, int cap) {
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kPpoThreads, 0) !=
          cudaSuccess ||
      per_sm < 1)
    per_sm = 1;
  const long long want = (work_items + kPpoThreads - 1) / kPpoThreads;
  long long g = static_cast<long long>(num_sms()) * per_sm;
  if (want < g) g = want;
  if (g > cap) g = cap;
  return g < 1 ? 1 : static_cast<int>(g);
}

struct WsLayout {
  MomPart* mom;
  LossPart* loss;
  double* moments;
  float* coef;
};

WsLayout layout(void* ws) {
  char* p = static_cast<char*>(ws);
  WsLayout w;
  w.mom = reinterpret_cast<MomPart*>(p);
  p += sizeof(MomPart) * kPpoMaxMomentBlocks;
  w.loss = reinterpret_cast<LossPart*>(p);
  p += sizeof(LossPart) * kPpoMaxLossBlocks;
  w.moments = reinterpret_cast<double*>(p);
  w.coef = reinterpret_cast<float*>(p + 4 * sizeof(double));
  return w;
}

bool vec4_ok(int64_t L, std::initializer_list<const void*> ptrs) {
  if (L % 4 != 0) return false;
  for (const void* p : ptrs)
    if (reinterpret_cast<uintptr_t>(p) % 16 != 0) return false;
  return true;
}

// Pass 1 and the coefficient merge. moments_out: where the fp64 moments go.
int launch_moments_coef(const float* adv, const int32_t* lengths, int S, int L, bool with_adv,
                        const double* ext, const WsLayout& w, double* moments_out, int* err,
                        cudaStream_t st) {
  int G = 0;
  if (ext == nullptr) {
    const bool v4 = vec4_ok(L, {adv});
    cudaError_t e;
    if (v4 && with_adv) {
      // a warp per row pair: S / 2 warps of work
      G = one_wave(ppo_moments_rows_kernel, (static_cast<long long>(S) + 1) / 2 * 32,
                   kPpoMaxMomentBlocks);
      e = launch_pdl(ppo_moments_rows_kernel, dim3(G), dim3(kPpoThreads), 0, st, adv, lengths, S,
                     L, w.mom, err);
    } else if (v4) {
      G = one_wave(ppo_moments_kernel<4>, S, kPpoMaxMomentBlocks);
      e = launch_pdl(ppo_moments_kernel<4>, dim3(G), dim3(kPpoThreads), 0, st, adv, lengths, S,
                     L, 0, w.mom, err);
    } else {
      G = one_wave(ppo_moments_kernel<1>, with_adv ? static_cast<long long>(S) * L : S,
                   kPpoMaxMomentBlocks);
      e = launch_pdl(ppo_moments_kernel<1>, dim3(G), dim3(kPpoThreads), 0, st, adv, lengths, S,
                     L, with_adv ? 1 : 0, w.mom, err);
    }
    if (e != cudaSuccess) return -3;
  }
  return launch_pdl(ppo_coef_kernel, dim3(1), dim3(kPpoThreads), 0, st, adv, S, L, with_adv ? 1 : 0,
                    static_cast<const MomPart*>(w.mom), G, ext, moments_out, w.coef) ==
                 cudaSuccess
             ? 0
             : -3;
}

}  // namespace

size_t ppo_loss_workspace_bytes() {
  return sizeof(MomPart) * kPpoMaxMomentBlocks + sizeof(LossPart) * kPpoMaxLossBlocks +
         4 * sizeof(double) + 4 * sizeof(float);
}

int launch_ppo_adv_moments(const float* adv, const int32_t* lengths, int64_t S, int64_t L,
                           double* out, void* ws, int* err, cudaStream_t st) {
  if (S * L == 0) {
    const WsLayout w = layout(ws);
    return launch_pdl(ppo_coef_kernel, dim3(1), dim3(kPpoThreads), 0, st, adv,
                      static_cast<int>(S), static_cast<int>(L), 0,
                      static_cast<const MomPart*>(w.mom), 0, static_cast<const double*>(nullptr),
                      out, w.coef) == cudaSuccess
               ? 0
               : -3;
  }
  return launch_moments_coef(adv, lengths, static_cast<int>(S), static_cast<int>(L), true,
                             nullptr, layout(ws), out, err, st);
}

int launch_ppo_loss(const float* logp_new, const float* logp_old, const float* adv,
                    const float* ret, const float* val, const int32_t* lengths, int64_t S,
                    int64_t L, float eps, bool whiten, const double* ext_moments,
                    float* grad_logp, float* grad_val, double* stats, void* ws, int* err,
                    cudaStream_t st) {
  const int Si = static_cast<int>(S), Li = static_cast<int>(L);
  const WsLayout w = layout(ws);
  const int report = (whiten || ext_moments != nullptr) ? 1 : 0;
  if (S * L == 0) {
    // empty batch: moments (the caller's, or none) and statistics only
    if (launch_pdl(ppo_coef_kernel, dim3(1), dim3(kPpoThreads), 0, st, adv, Si, Li, 0,
                   static_cast<const MomPart*>(w.mom), 0, ext_moments, w.moments, w.coef) !=
        cudaSuccess)
      return -3;
    return launch_pdl(ppo_finalize_kernel, dim3(1), dim3(kPpoThreads), 0, st,
                      static_cast<const LossPart*>(w.loss), 0,
                      static_cast<const double*>(w.moments), report, stats) == cudaSuccess
               ? 0
               : -3;
  }
  if (launch_moments_coef(adv, lengths, Si, Li, whiten, ext_moments, w, w.moments, err, st) != 0)
    return -3;
  const bool v4 = vec4_ok(L, {logp_new, logp_old, adv, ret, val, grad_logp, grad_val});
  const long long items = S * (v4 ? L / 4 : L);
  int G = 0;
  cudaError_t e;
#define HY_PPO_LAUNCH(V, W)                                                                      \
  G = one_wave(ppo_loss_kernel<V, W>, items, kPpoMaxLossBlocks);                                \
  e = launch_pdl(ppo_loss_kernel<V, W>, dim3(G), dim3(kPpoThreads), 0, st, logp_new, logp_old, \
                 adv, ret, val, lengths, Si, Li, eps, static_cast<const float*>(w.coef), w.loss, \
                 grad_logp, grad_val, err)
  if (v4) {
    if (whiten) { HY_PPO_LAUNCH(4, true); } else { HY_PPO_LAUNCH(4, false); }
  } else {
    if (whiten) { HY_PPO_LAUNCH(1, true); } else { HY_PPO_LAUNCH(1, false); }
  }
#undef HY_PPO_LAUNCH
  if (e != cudaSuccess) return -3;
  return launch_pdl(ppo_finalize_kernel, dim3(1), dim3(kPpoThreads), 0, st,
                    static_cast<const LossPart*>(w.loss), G,
                    static_cast<const double*>(w.moments), report, stats) == cudaSuccess
             ? 0
             : -3;
}

}  // namespace hydra
