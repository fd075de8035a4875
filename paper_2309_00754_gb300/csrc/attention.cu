// Causal self-attention of the Llama decoder in the full scoring pass (the paper runs
// Llama 7b, §4), for both streams at once (each stream's sequences are separate rows):
//     o = softmax(q k^T / sqrt(Dh) + causal mask) v,   head dim Dh = 128
// q, k, v are the column blocks [0, d), [d, 2d), [2d, 3d) of the fused projection output
// (row stride ld); o is written to columns [h Dh, (h + 1) Dh) of out.
//
// One CTA (4 warps) per 64 queries of one (sequence, head); each warp owns 16 query rows.
// Keys and values stream in 64-row blocks, double-buffered with cp.async into XOR-swizzled
// shared memory; q k^T and p v run on mma.sync m16n8k16 (bf16 in, fp32 accumulate) with an
// online softmax (running max and sum per row) in registers, so the score matrix never
// leaves the SM. The probabilities enter p v as a bf16 hi/lo pair (two MMAs), so they keep
// about 16 mantissa bits instead of bf16's 8. Attention is about 1.5 % of the pass's flops;
// the projections run on the tcgen05 kernel.
#include <float.h>

#include "common.cuh"
#include "kernels.h"

namespace hydra {
namespace {

constexpr int kDh = 128;
constexpr int kBM = 64;  // queries per CTA
constexpr int kBN = 64;  // keys per block
constexpr int kThreads = 128;
constexpr int kTileBytes = kBM * kDh * 2;  // 16 KiB
constexpr int kSmem = kTileBytes * 5;      // Q + 2 x (K, V)

// byte offset of 16-byte chunk `ch` (0..15) of row `row` in a [rows x 256 B] tile
__device__ __forceinline__ uint32_t swz(int row, int ch) {
  return static_cast<uint32_t>(row * 256 + ((ch ^ (row & 7)) << 4));
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool ok) {
  const int n = ok ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n)
               : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& a, uint32_t& b, uint32_t& c,
                                        uint32_t& d) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(a), "=r"(b), "=r"(c), "=r"(d)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& a, uint32_t& b, uint32_t& c,
                                          uint32_t& d) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(a), "=r"(b), "=r"(c), "=r"(d)
               : "r"(addr));
}

__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// copy rows [row0, row0 + 64) (clipped at P) of one 128-column block into a swizzled tile
__device__ __forceinline__ void load_tile(uint32_t tile, const __nv_bfloat16* base, int row0, int P,
                                          int ld) {
  for (int e = threadIdx.x; e < kBM * 16; e += kThreads) {
    const int row = e >> 4, ch = e & 15;
    const bool ok = row0 + row < P;
    const __nv_bfloat16* src = base + static_cast<size_t>(ok ? row0 + row : 0) * ld + ch * 8;
    cp_async16(tile + swz(row, ch), src, ok);
  }
}

__global__ void __launch_bounds__(kThreads)
    causal_attention_kernel(const __nv_bfloat16* __restrict__ qkv, int P, int ld, int d,
                            float scale_log2, __nv_bfloat16* __restrict__ out, int ld_out) {
  extern __shared__ __align__(1024) uint8_t smem[];
  const int nqb = (P + kBM - 1) / kBM;
  const int qb = nqb - 1 - static_cast<int>(blockIdx.x);  // longest rows first
  const int head = blockIdx.y;
  const int seq = blockIdx.z;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int g = lane >> 2, c = lane & 3;

  const __nv_bfloat16* qbase = qkv + static_cast<size_t>(seq) * P * ld + head * kDh;
  const __nv_bfloat16* kbase = qbase + d;
  const __nv_bfloat16* vbase = qbase + 2 * d;
  const uint32_t sQ = smem_u32(smem);
  const uint32_t sK[2] = {sQ + kTileBytes, sQ + 3 * kTileBytes};
  const uint32_t sV[2] = {sQ + 2 * kTileBytes, sQ + 4 * kTileBytes};

  load_tile(sQ, qbase, qb * kBM, P, ld);
  cp_commit();
  load_tile(sK[0], kbase, 0, P, ld);
  load_tile(sV[0], vbase, 0, P, ld);
  cp_commit();

  cp_wait<1>();
  __syncthreads();
  // Q fragments of this warp's 16 rows: 8 k-steps of 16 dims
  uint32_t qf[8][4];
#pragma unroll
  for (int kk = 0; kk < 8; ++kk) {
    const int row = warp * 16 + (lane & 15);
    const int ch = 2 * kk + (lane >> 4);
    ldsm_x4(sQ + swz(row, ch), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
  }

  float o[16][4];
#pragma unroll
  for (int n = 0; n < 16; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
  float m_lo = -FLT_MAX, m_hi = -FLT_MAX, l_lo = 0.f, l_hi = 0.f;
  const int q_lo = qb * kBM + warp * 16 + g;  // query index of rows g and g + 8
  const int q_hi = q_lo + 8;

  for (int j = 0; j <= qb; ++j) {
    const int st = j & 1;
    if (j < qb) {
      load_tile(sK[st ^ 1], kbase, (j + 1) * kBN, P, ld);
      load_tile(sV[st ^ 1], vbase, (j + 1) * kBN, P, ld);
      cp_commit();
      cp_wait<1>();
    } else {
      cp_wait<0>();
    }
    __syncthreads();

    // scores for 64 keys: 8 n-tiles of 8 keys
    float s[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
      for (int kk = 0; kk < 8; kk += 2) {
        // matrices: keys nt*8 + (lane & 7), dims (kk*16 + (lane >> 3) * 8)
        uint32_t b0, b1, b2, b3;
        const int row = nt * 8 + (lane & 7);
        const int ch = 2 * kk + (lane >> 3);
        ldsm_x4(sK[st] + swz(row, ch), b0, b1, b2, b3);
        mma16816(s[nt], qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3], b0, b1);
        mma16816(s[nt], qf[kk + 1][0], qf[kk + 1][1], qf[kk + 1][2], qf[kk + 1][3], b2, b3);
      }
    }
    // scale (log2 domain) and causal mask on the diagonal block
    float mx_lo = -FLT_MAX, mx_hi = -FLT_MAX;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int key = j * kBN + nt * 8 + 2 * c + e;
        float a = s[nt][e] * scale_log2;
        float b = s[nt][2 + e] * scale_log2;
        if (key > q_lo) a = -FLT_MAX;
        if (key > q_hi) b = -FLT_MAX;
        s[nt][e] = a;
        s[nt][2 + e] = b;
        mx_lo = fmaxf(mx_lo, a);
        mx_hi = fmaxf(mx_hi, b);
      }
    }
#pragma unroll
    for (int off = 1; off <= 2; off <<= 1) {
      mx_lo = fmaxf(mx_lo, __shfl_xor_sync(0xffffffffu, mx_lo, off));
      mx_hi = fmaxf(mx_hi, __shfl_xor_sync(0xffffffffu, mx_hi, off));
    }
    const float mn_lo = fmaxf(m_lo, mx_lo), mn_hi = fmaxf(m_hi, mx_hi);
    const float corr_lo = exp2f(m_lo - mn_lo), corr_hi = exp2f(m_hi - mn_hi);
    m_lo = mn_lo;
    m_hi = mn_hi;
    float sum_lo = 0.f, sum_hi = 0.f;
    // probabilities as bf16 pairs [n-tile][row g / row g+8], split p = hi + lo so that the
    // p v product keeps ~16 mantissa bits of p (one bf16 operand alone keeps 8)
    uint32_t pf[8][2], pl[8][2];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const float p0 = exp2f(s[nt][0] - mn_lo), p1 = exp2f(s[nt][1] - mn_lo);
      const float p2 = exp2f(s[nt][2] - mn_hi), p3 = exp2f(s[nt][3] - mn_hi);
      sum_lo += p0 + p1;
      sum_hi += p2 + p3;
      pf[nt][0] = pack_bf16x2(p0, p1);
      pf[nt][1] = pack_bf16x2(p2, p3);
      const float2 h01 = unpack_bf16x2(pf[nt][0]), h23 = unpack_bf16x2(pf[nt][1]);
      pl[nt][0] = pack_bf16x2(p0 - h01.x, p1 - h01.y);
      pl[nt][1] = pack_bf16x2(p2 - h23.x, p3 - h23.y);
    }
    l_lo = l_lo * corr_lo + sum_lo;
    l_hi = l_hi * corr_hi + sum_hi;
#pragma unroll
    for (int n = 0; n < 16; ++n) {
      o[n][0] *= corr_lo;
      o[n][1] *= corr_lo;
      o[n][2] *= corr_hi;
      o[n][3] *= corr_hi;
    }
    // o += (p_hi + p_lo) v: k-steps of 16 keys, n-tiles of 8 dims
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      const uint32_t a0 = pf[2 * kk][0], a1 = pf[2 * kk][1];
      const uint32_t a2 = pf[2 * kk + 1][0], a3 = pf[2 * kk + 1][1];
      const uint32_t c0 = pl[2 * kk][0], c1 = pl[2 * kk][1];
      const uint32_t c2 = pl[2 * kk + 1][0], c3 = pl[2 * kk + 1][1];
#pragma unroll
      for (int n = 0; n < 16; n += 2) {
        // matrices: keys kk*16 + (i & 1) * 8 + (lane & 7), dims n*8 + (i >> 1) * 8
        const int i = lane >> 3;
        const int row = kk * 16 + (i & 1) * 8 + (lane & 7);
        const int ch = n + (i >> 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(sV[st] + swz(row, ch), b0, b1, b2, b3);
        mma16816(o[n], a0, a1, a2, a3, b0, b1);
        mma16816(o[n + 1], a0, a1, a2, a3, b2, b3);
        mma16816(o[n], c0, c1, c2, c3, b0, b1);
        mma16816(o[n + 1], c0, c1, c2, c3, b2, b3);
      }
    }
    __syncthreads();
  }

  // normalise and store this warp's 16 rows
#pragma unroll
  for (int off = 1; off <= 2; off <<= 1) {
    l_lo += __shfl_xor_sync(0xffffffffu, l_lo, off);
    l_hi += __shfl_xor_sync(0xffffffffu, l_hi, off);
  }
  const float inv_lo = 1.f / l_lo, inv_hi = 1.f / l_hi;
  __nv_bfloat16* obase = out + static_cast<size_t>(seq) * P * ld_out + head * kDh;
#pragma unroll
  for (int n = 0; n < 16; ++n) {
    const int col = n * 8 + 2 * c;
    if (q_lo < P)
      *reinterpret_cast<uint32_t*>(obase + static_cast<size_t>(q_lo) * ld_out + col) =
          pack_bf16x2(o[n][0] * inv_lo, o[n][1] * inv_lo);
    if (q_hi < P)
      *reinterpret_cast<uint32_t*>(obase + static_cast<size_t>(q_hi) * ld_out + col) =
          pack_bf16x2(o[n][2] * inv_hi, o[n][3] * inv_hi);
  }
}

}  // namespace

int launch_causal_attention(const void* qkv, int64_t nseq, int64_t P, int64_t ld, int64_t n_heads,
                            int64_t head_dim, void* out, int64_t ld_out, cudaStream_t st) {
  if (nseq == 0 || P == 0) return 0;
  if (head_dim != kDh) return -4;
  static bool attr_set = false;
  if (!attr_set) {
    if (cudaFuncSetAttribute(causal_attention_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kSmem) != cudaSuccess)
      return -1;
    attr_set = true;
  }
  const int nqb = static_cast<int>((P + kBM - 1) / kBM);
  const dim3 grid(nqb, static_cast<unsigned>(n_heads), static_cast<unsigned>(nseq));
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(head_dim));
  causal_attention_kernel<<<grid, kThreads, kSmem, st>>>(
      static_cast<const __nv_bfloat16*>(qkv), static_cast<int>(P), static_cast<int>(ld),
      static_cast<int>(n_heads * head_dim), scale_log2, static_cast<__nv_bfloat16*>(out),
      static_cast<int>(ld_out));
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace hydra
