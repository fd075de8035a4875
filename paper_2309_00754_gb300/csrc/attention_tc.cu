// Causal self-attention of the Llama decoder on the 5th-generation tensor cores (tcgen05 +
// TMEM + TMA), for both streams at once (each stream's sequences are separate rows):
//     o = softmax(q k^T / sqrt(Dh) + causal mask) v,   head dim Dh = 128
// q, k, v are the column blocks [0, d), [d, 2d), [2d, 3d) of the fused projection output
// (row stride ld); o is written to columns [h Dh, (h + 1) Dh) of out.
//
// One CTA per 128 queries of one (sequence, head), key/value blocks of 128 rows, flash
// attention with an online softmax:
//  * warp 0 moves Q once and each K / V block through a 2-stage ring with TMA (128-byte
//    swizzle, [128 rows x 64] boxes);
//  * warp 1 owns TMEM and issues tcgen05.mma from one elected lane: S_j = Q K_j^T into one of
//    two fp32 S accumulators (so Q K_{j+1}^T runs while the softmax works on S_j), then
//    O += P_j V_j into the O accumulator, with V read as an MN-major operand;
//  * warps 2..5 are the softmax: thread i owns query row i (TMEM lane i), so row maxima and
//    sums need no shuffles. P_j goes to shared memory as bf16 in the 128-byte-swizzled
//    K-major layout the P V MMA reads. The running maximum is a reference value that moves
//    only when a row's maximum grows by more than 2^8 (then the thread rescales its O row in
//    TMEM); O and the row sum l share the reference, so O / l is exact either way and every
//    p stays at most 2^8. After the last block each thread normalises its O row and stores it.
// The probabilities enter P V as bf16 (8 mantissa bits); l sums the same rounded values, so
// each output row is an exact convex combination of v rows with weights within 2^-9 of p.
#include <float.h>

#include "common.cuh"
#include "kernels.h"

namespace hydra {
namespace attn_tc {

constexpr int kDh = 128;
constexpr int kBQ = 128;                    // queries per CTA (MMA M, TMEM lanes)
constexpr int kBK = 128;                    // keys per block
constexpr int kThreads = 192;               // producer, MMA, 4 softmax warps
constexpr int kTile = 128 * 64 * 2;         // [128 rows x 64 bf16] swizzled tile: 16 KiB
constexpr int kMat = 2 * kTile;             // [128 x 128] bf16 operand: 32 KiB
constexpr int kOffQ = 0;
constexpr int kOffK = kOffQ + kMat;         // 2 stages
constexpr int kOffV = kOffK + 2 * kMat;     // 2 stages
constexpr int kOffP = kOffV + 2 * kMat;
constexpr int kOffBar = kOffP + kMat;
constexpr int kNumBars = 14;
constexpr int kSmem = 1024 + kOffBar + kNumBars * 8 + 16;
constexpr uint32_t kTmemCols = 512;         // S0 [0,128), S1 [128,256), O [256,384)
constexpr uint32_t kColO = 256;

// instruction descriptors (kind::f16, bf16 A/B, fp32 D): S = Q K^T (both K-major) and
// O += P V with V MN-major (bit 16)
constexpr uint32_t kIdescQK = idesc_bf16_f32(kBQ, kBK);
constexpr uint32_t kIdescPV = idesc_bf16_f32(kBQ, kDh) | (1u << 16);

// Shared-memory descriptor of an MN-major bf16 operand stored as [K rows x 64] tiles with
// 128-byte swizzle (TMA boxes of 64 MN elements by K rows): 64 MN elements per 128-byte row,
// K rows 128 B apart, 8-row groups 1024 B apart (stride byte offset), the next 64 MN
// elements one tile (`mn_stride` bytes) further (leading byte offset).
__device__ __forceinline__ uint64_t smem_desc_sw128_mn(uint32_t addr, uint32_t mn_stride) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((addr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>((mn_stride >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>(1024u >> 4) << 32;
  d |= static_cast<uint64_t>(1u) << 46;
  d |= static_cast<uint64_t>(2u) << 61;
  return d;
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// 32 lanes x 64 consecutive 32-bit columns: thread i of the warp receives lane (base + i)
__device__ __forceinline__ void tc_ld_x64(uint32_t taddr, float (&r)[64]) {
  uint32_t (&u)[64] = reinterpret_cast<uint32_t(&)[64]>(r);
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x64.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,"
      "%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,"
      "%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, [%64];"
      : "=r"(u[0]), "=r"(u[1]), "=r"(u[2]), "=r"(u[3]), "=r"(u[4]), "=r"(u[5]), "=r"(u[6]),
        "=r"(u[7]), "=r"(u[8]), "=r"(u[9]), "=r"(u[10]), "=r"(u[11]), "=r"(u[12]), "=r"(u[13]),
        "=r"(u[14]), "=r"(u[15]), "=r"(u[16]), "=r"(u[17]), "=r"(u[18]), "=r"(u[19]),
        "=r"(u[20]), "=r"(u[21]), "=r"(u[22]), "=r"(u[23]), "=r"(u[24]), "=r"(u[25]),
        "=r"(u[26]), "=r"(u[27]), "=r"(u[28]), "=r"(u[29]), "=r"(u[30]), "=r"(u[31]),
        "=r"(u[32]), "=r"(u[33]), "=r"(u[34]), "=r"(u[35]), "=r"(u[36]), "=r"(u[37]),
        "=r"(u[38]), "=r"(u[39]), "=r"(u[40]), "=r"(u[41]), "=r"(u[42]), "=r"(u[43]),
        "=r"(u[44]), "=r"(u[45]), "=r"(u[46]), "=r"(u[47]), "=r"(u[48]), "=r"(u[49]),
        "=r"(u[50]), "=r"(u[51]), "=r"(u[52]), "=r"(u[53]), "=r"(u[54]), "=r"(u[55]),
        "=r"(u[56]), "=r"(u[57]), "=r"(u[58]), "=r"(u[59]), "=r"(u[60]), "=r"(u[61]),
        "=r"(u[62]), "=r"(u[63])
      : "r"(taddr)
      : "memory");
}

// 32 lanes x 32 consecutive 32-bit columns from registers: thread i writes lane (base + i)
__device__ __forceinline__ void tc_st_x32(uint32_t taddr, const uint32_t (&u)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(u[0]), "r"(u[1]), "r"(u[2]), "r"(u[3]), "r"(u[4]), "r"(u[5]), "r"(u[6]), "r"(u[7]),
      "r"(u[8]), "r"(u[9]), "r"(u[10]), "r"(u[11]), "r"(u[12]), "r"(u[13]), "r"(u[14]),
      "r"(u[15]), "r"(u[16]), "r"(u[17]), "r"(u[18]), "r"(u[19]), "r"(u[20]), "r"(u[21]),
      "r"(u[22]), "r"(u[23]), "r"(u[24]), "r"(u[25]), "r"(u[26]), "r"(u[27]), "r"(u[28]),
      "r"(u[29]), "r"(u[30]), "r"(u[31])
      : "memory");
}

__device__ __forceinline__ void tc_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c,
                                             uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c),
               "r"(d)
               : "memory");
}

__global__ void __launch_bounds__(kThreads, 1)
    causal_attention_tc_kernel(const __grid_constant__ CUtensorMap tm_qkv, int P, int d,
                               float scale_log2, __nv_bfloat16* __restrict__ out, int ld_out,
                               int* err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kOffBar);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + kNumBars);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int nqb = (P + kBQ - 1) / kBQ;
  const int qb = nqb - 1 - static_cast<int>(blockIdx.x);  // longest rows first
  const int head = blockIdx.y;
  const int seq = blockIdx.z;
  const int nblk = qb + 1;                                 // causal: key blocks 0..qb
  const int row0 = seq * P;                                // first row of this sequence

  const uint32_t sbase = smem_u32(smem);
  const uint32_t sQ = sbase + kOffQ, sK = sbase + kOffK, sV = sbase + kOffV, sP = sbase + kOffP;
  auto bar = [&](int i) { return smem_u32(&bars[i]); };
  const uint32_t q_full = bar(0);
  auto k_full = [&](int b) { return bar(1 + b); };
  auto v_full = [&](int b) { return bar(3 + b); };
  auto kv_empty = [&](int b) { return bar(5 + b); };
  auto s_full = [&](int b) { return bar(7 + b); };
  auto s_free = [&](int b) { return bar(9 + b); };
  const uint32_t p_full = bar(11);
  const uint32_t pv_done = bar(12);
  const uint32_t mma_done = bar(13);

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(k_full(b), 1);
      mbar_init(v_full(b), 1);
      mbar_init(kv_empty(b), 1);
      mbar_init(s_full(b), 1);
      mbar_init(s_free(b), 4);
    }
    mbar_init(p_full, 4);
    mbar_init(pv_done, 1);
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (elect_one()) {
      tma_prefetch_desc(&tm_qkv);
      mbar_arrive_expect_tx(q_full, kMat);
      const int y = row0 + qb * kBQ;
      tma_load_2d(sQ, &tm_qkv, head * kDh, y, q_full);
      tma_load_2d(sQ + kTile, &tm_qkv, head * kDh + 64, y, q_full);
    }
    __syncwarp();
    int issued = 0;
    for (int j = 0; j < nblk; ++j) {
      const int b = j & 1;
      if (j >= 2 && !warp_wait_bounded(kv_empty(b), ((j - 2) >> 1) & 1, abort_flag, err,
                                       kDevTimeoutProducer))
        break;
      if (elect_one()) {
        const int y = row0 + j * kBK;
        mbar_arrive_expect_tx(k_full(b), kMat);
        tma_load_2d(sK + b * kMat, &tm_qkv, d + head * kDh, y, k_full(b));
        tma_load_2d(sK + b * kMat + kTile, &tm_qkv, d + head * kDh + 64, y, k_full(b));
        mbar_arrive_expect_tx(v_full(b), kMat);
        tma_load_2d(sV + b * kMat, &tm_qkv, 2 * d + head * kDh, y, v_full(b));
        tma_load_2d(sV + b * kMat + kTile, &tm_qkv, 2 * d + head * kDh + 64, y, v_full(b));
      }
      __syncwarp();
      issued = j + 1;
    }
    // copies in flight land before the CTA's shared memory is released
    volatile int no_abort = 0;
    warp_wait_bounded(q_full, 0, &no_abort, err, kDevTimeoutDrain);
    for (int j = (issued > 2 ? issued - 2 : 0); j < issued; ++j) {
      warp_wait_bounded(k_full(j & 1), (j >> 1) & 1, &no_abort, err, kDevTimeoutDrain);
      warp_wait_bounded(v_full(j & 1), (j >> 1) & 1, &no_abort, err, kDevTimeoutDrain);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    bool ok = warp_wait_bounded(q_full, 0, abort_flag, err, kDevTimeoutMma);
    // S_j = Q K_j^T into S accumulator j & 1
    auto issue_s = [&](int j) {
      const int b = j & 1;
      if (!warp_wait_bounded(k_full(b), (j >> 1) & 1, abort_flag, err, kDevTimeoutMma)) return false;
      if (j >= 2 &&
          !warp_wait_bounded(s_free(b), ((j - 2) >> 1) & 1, abort_flag, err, kDevTimeoutMma))
        return false;
      tc_fence_after();
      if (elect_one()) {
        const uint32_t kb = sK + b * kMat;
#pragma unroll
        for (int k = 0; k < kDh / 16; ++k) {
          const uint32_t off = (k >> 2) * kTile + (k & 3) * 32;
          tc_mma_bf16(tmem + b * kBK, smem_desc_sw128(sQ + off), smem_desc_sw128(kb + off),
                      kIdescQK, k > 0 ? 1u : 0u);
        }
        tc_commit(s_full(b));
      }
      __syncwarp();
      return true;
    };
    if (ok) ok = issue_s(0);
    for (int j = 0; j < nblk && ok; ++j) {
      const int b = j & 1;
      if (j + 1 < nblk && !issue_s(j + 1)) break;
      // O += P_j V_j once the softmax has written P_j
      if (!warp_wait_bounded(p_full, j & 1, abort_flag, err, kDevTimeoutMma) ||
          !warp_wait_bounded(v_full(b), (j >> 1) & 1, abort_flag, err, kDevTimeoutMma))
        break;
      tc_fence_after();
      if (elect_one()) {
        const uint32_t vb = sV + b * kMat;
#pragma unroll
        for (int k = 0; k < kBK / 16; ++k) {
          // A: P keys [16k, 16k + 16) (K-major); B: V rows [16k, 16k + 16) (MN-major)
          const uint32_t poff = (k >> 2) * kTile + (k & 3) * 32;
          tc_mma_bf16(tmem + kColO, smem_desc_sw128(sP + poff),
                      smem_desc_sw128_mn(vb + k * 2048, kTile), kIdescPV,
                      (j > 0 || k > 0) ? 1u : 0u);
        }
        tc_commit(pv_done);
        tc_commit(kv_empty(b));
      }
      __syncwarp();
    }
    // every issued MMA has finished before TMEM is released
    if (elect_one()) tc_commit(mma_done);
    __syncwarp();
    volatile int no_abort = 0;
    warp_wait_bounded(mma_done, 0, &no_abort, err, kDevTimeoutDrain);
  } else {
    // ---------------------------------------------------------------- softmax (4 warps)
    const int q4 = warp & 3;                  // this warp may access TMEM lanes [32 q4, +32)
    const int row = q4 * 32 + lane;           // query row of the block = TMEM lane
    const int q = qb * kBQ + row;             // query position in the sequence
    const uint32_t t_lane = tmem + (static_cast<uint32_t>(q4 * 32) << 16);
    float m_ref = -FLT_MAX;                   // reference maximum, log2 domain
    float l = 0.f;                            // sum of the (bf16-rounded) probabilities
    bool ok = true;
    for (int j = 0; j < nblk; ++j) {
      const int b = j & 1;
      if (!warp_wait_bounded(s_full(b), (j >> 1) & 1, abort_flag, err, kDevTimeoutEpilogue)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float s[kBK];
      tc_ld_x64(t_lane + b * kBK, *reinterpret_cast<float(*)[64]>(s));
      tc_ld_x64(t_lane + b * kBK + 64, *reinterpret_cast<float(*)[64]>(s + 64));
      tc_wait_ld();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(s_free(b));  // S_j is in registers: the buffer may be reused
      // log2-domain scores; on the diagonal block key c is visible to row `row` iff c <= row
      const int kmax = (j == qb) ? row : kBK - 1;
      float mx = -FLT_MAX;
#pragma unroll
      for (int c = 0; c < kBK; ++c) {
        const float x = c <= kmax ? s[c] * scale_log2 : -INFINITY;
        s[c] = x;
        mx = fmaxf(mx, x);
      }
      bool rescale = false;
      float corr = 1.f;
      if (j == 0) {
        m_ref = mx;
      } else if (mx > m_ref + 8.f) {
        corr = ex2(m_ref - mx);
        m_ref = mx;
        rescale = true;
      }
      // P_{j-1} V_{j-1} has finished: the P buffer is free and O is stable
      if (j > 0 && !warp_wait_bounded(pv_done, (j - 1) & 1, abort_flag, err, kDevTimeoutEpilogue)) {
        ok = false;
        break;
      }
      tc_fence_after();
      if (__any_sync(0xffffffffu, rescale)) {
        l *= corr;
#pragma unroll 1
        for (int h = 0; h < 4; ++h) {
          uint32_t o[32];
          tc_ld_32x32b_x32(t_lane + kColO + 32 * h, o);
          tc_wait_ld();
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * corr);
          tc_st_x32(t_lane + kColO + 32 * h, o);
        }
        tc_wait_st();
      }
      // P_j = 2^(s - m_ref) as bf16 into the swizzled K-major P tile (row `row`)
      float sum = 0.f;
#pragma unroll
      for (int ch = 0; ch < kBK / 8; ++ch) {
        uint32_t w[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          w[e] = pack_bf16x2(ex2(s[8 * ch + 2 * e] - m_ref), ex2(s[8 * ch + 2 * e + 1] - m_ref));
          const float2 r = unpack_bf16x2(w[e]);
          sum += r.x + r.y;
        }
        const uint32_t addr = sP + (ch >> 3) * kTile + row * 128 + (((ch & 7) ^ (row & 7)) << 4);
        st_shared_v4(addr, w[0], w[1], w[2], w[3]);
      }
      l += sum;
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // visible to the MMA
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full);
    }
    // normalise and store this thread's output row
    if (ok && warp_wait_bounded(pv_done, (nblk - 1) & 1, abort_flag, err, kDevTimeoutEpilogue)) {
      tc_fence_after();
      const float inv = 1.f / l;
      __nv_bfloat16* orow = out + static_cast<size_t>(row0 + q) * ld_out + head * kDh;
#pragma unroll 1
      for (int h = 0; h < 4; ++h) {
        uint32_t o[32];
        tc_ld_32x32b_x32(t_lane + kColO + 32 * h, o);
        tc_wait_ld();
        if (q < P) {
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            auto f = [&](int e) { return __uint_as_float(o[8 * i + e]) * inv; };
            uint4 v;
            v.x = pack_bf16x2(f(0), f(1));
            v.y = pack_bf16x2(f(2), f(3));
            v.z = pack_bf16x2(f(4), f(5));
            v.w = pack_bf16x2(f(6), f(7));
            *reinterpret_cast<uint4*>(orow + 32 * h + 8 * i) = v;
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace attn_tc

int launch_causal_attention(const void* qkv, int64_t nseq, int64_t P, int64_t ld, int64_t n_heads,
                            int64_t head_dim, void* out, int64_t ld_out, cudaStream_t st) {
  using namespace attn_tc;
  if (nseq == 0 || P == 0) return 0;
  if (head_dim != kDh) return -4;
  static bool attr_set = false;
  if (!attr_set) {
    if (cudaFuncSetAttribute(causal_attention_tc_kernel,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem) != cudaSuccess)
      return -1;
    attr_set = true;
  }
  int* err = device_error_word();
  if (err == nullptr) return -1;
  const int64_t d = n_heads * head_dim;
  CUtensorMap map;
  if (!make_tma_map(&map, qkv, nseq * P, 3 * d, ld, 128, false)) return -2;
  const int nqb = static_cast<int>((P + kBQ - 1) / kBQ);
  const dim3 grid(nqb, static_cast<unsigned>(n_heads), static_cast<unsigned>(nseq));
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(head_dim));
  causal_attention_tc_kernel<<<grid, kThreads, kSmem, st>>>(
      map, static_cast<int>(P), static_cast<int>(d), scale_log2, static_cast<__nv_bfloat16*>(out),
      static_cast<int>(ld_out), err);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace hydra
