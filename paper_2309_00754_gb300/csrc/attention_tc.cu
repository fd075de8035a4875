// Causal self-attention of the Llama decoder on the 5th-generation tensor cores (tcgen05 +
// TMEM + TMA), for both streams at once (each stream's sequences are separate rows):
//     o = softmax(q k^T / sqrt(Dh) + causal mask) v,   head dim Dh = 128
// q, k, v are the column blocks [0, d), [d, 2d), [2d, 3d) of the fused projection output
// (row stride ld); o is written to columns [h Dh, (h + 1) Dh) of out.
//
// Persistent CTAs (one per SM) take tiles of 128 queries of one (sequence, head), longest
// first; key/value blocks of 128 rows; flash attention with an online softmax. The rings
// run on across tiles, so the next tile's loads and first Q K^T overlap this tile's tail:
//  * warp 0 moves Q per tile and the K / V blocks through 3-stage rings with TMA (128-byte
//    swizzle, [128 rows x 64] boxes); a K stage is released as soon as its Q K^T is done;
//  * warp 1 owns TMEM and issues tcgen05.mma from one elected lane: S_j = Q K_j^T into the
//    fp32 S accumulator, which the softmax copies to registers at once, so Q K_{j+1}^T runs
//    while the softmax works on S_j; then O += P_j V_j into one of two O accumulators (one
//    per tile in flight), with P read from TMEM and V as an MN-major shared-memory operand;
//  * warps 2..5 are the softmax: thread i owns query row i (TMEM lane i), so row maxima and
//    sums need no shuffles. P_j is computed in registers (overlapping P_{j-1} V_{j-1}) and
//    stored to TMEM as bf16 pairs, so it costs no shared-memory bandwidth: the operand
//    traffic left in shared memory (K and V in, Q K^T and P V operand reads) is what bounds
//    a block. The running maximum is a reference value that moves
//    only when a row's maximum grows by more than 2^8 (then the thread rescales its O row in
//    TMEM); O and the row sum l share the reference, so O / l is exact either way and every
//    p stays at most 2^8;
//  * warps 6..9 are the epilogue: once a tile's last P V is done they normalise its O rows
//    by the row sums the softmax left in shared memory and store them.
// The probabilities enter P V as bf16 (8 mantissa bits, relative error at most 2^-9); the row
// sum l accumulates them in fp32.
#include <float.h>

#include "common.cuh"
#include "kernels.h"

namespace hydra {
namespace attn_tc {

constexpr int kDh = 128;
constexpr int kBQ = 128;                    // queries per CTA (MMA M, TMEM lanes)
constexpr int kBK = 128;                    // keys per block
constexpr int kThreads = 320;               // producer, MMA, 4 softmax, 4 epilogue warps
constexpr int kTile = 128 * 64 * 2;         // [128 rows x 64 bf16] swizzled tile: 16 KiB
constexpr int kMat = 2 * kTile;             // [128 x 128] bf16 operand: 32 KiB
constexpr int kOffQ = 0;
constexpr int kKStages = 3;                 // K ring: K_{j+3} loads once Q K_j^T is done
constexpr int kVStages = 3;                 // V ring: V_{j+3} loads once P_j V_j is done
constexpr int kOffK = kOffQ + kMat;
constexpr int kOffV = kOffK + kKStages * kMat;
constexpr int kOffL = kOffV + kVStages * kMat;  // final row sums of two tiles: 2 x 128 fp32
constexpr int kOffBar = kOffL + 2 * kBQ * 4;
constexpr int kNumBars = 25;
constexpr int kSmem = 1024 + kOffBar + kNumBars * 8 + 16;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS = 0;               // S: 128 fp32 columns
constexpr uint32_t kColP = 128;             // P: 128 bf16 = 64 columns
constexpr uint32_t kColO = 256;             // O0, O1: 128 fp32 columns each

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

// D[tmem] (+)= A[tmem] * B[smem]^T, bf16 inputs, fp32 accumulation: A is M rows (TMEM lanes)
// by K = 16 elements, two bf16 per 32-bit column (8 columns from a_tmem)
__device__ __forceinline__ void tc_mma_ts_bf16(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                               uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}


// This CTA's work: tiles t = blockIdx.x + i * gridDim.x (i = 0, 1, ...) of the ordering
// t -> (query block qb, head, sequence) with the largest qb (most key blocks) first, so the
// static round-robin assignment stays balanced; each tile runs key blocks j = 0..qb.
struct BlockCursor {
  int nqb, heads, nseq, ntiles, stride;
  int t, i, j;        // tile, this CTA's tile number, key block
  int qb, head, seq;  // decoded tile
  __device__ void init(int nqb_, int heads_, int nseq_, int first, int step) {
    nqb = nqb_;
    heads = heads_;
    nseq = nseq_;
    ntiles = nqb * heads * nseq;
    stride = step;
    t = first;
    i = 0;
    j = 0;
    decode();
  }
  __device__ void decode() {
    if (t >= ntiles) return;
    const int hs = heads * nseq;
    qb = nqb - 1 - t / hs;
    const int r = t % hs;
    head = r % heads;
    seq = r / heads;
  }
  __device__ bool valid() const { return t < ntiles; }
  __device__ bool last() const { return j == qb; }
  __device__ void next() {
    if (++j > qb) {
      j = 0;
      ++i;
      t += stride;
      decode();
    }
  }
};

__global__ void __launch_bounds__(kThreads, 1)
    causal_attention_tc_kernel(const __grid_constant__ CUtensorMap tm_qkv, int P, int d,
                               int n_heads, int nseq, float scale_log2,
                               __nv_bfloat16* __restrict__ out, int ld_out, int* err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  float* l_sm = reinterpret_cast<float*>(smem + kOffL);  // [2][kBQ]
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kOffBar);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + kNumBars);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int nqb = (P + kBQ - 1) / kBQ;

  const uint32_t sbase = smem_u32(smem);
  const uint32_t sQ = sbase + kOffQ, sK = sbase + kOffK, sV = sbase + kOffV;
  auto bar = [&](int i) { return smem_u32(&bars[i]); };
  const uint32_t q_full = bar(0);
  const uint32_t q_empty = bar(1);
  auto k_full = [&](int i) { return bar(2 + i); };
  auto k_empty = [&](int i) { return bar(5 + i); };
  auto v_full = [&](int i) { return bar(8 + i); };
  auto v_empty = [&](int i) { return bar(11 + i); };
  const uint32_t s_full = bar(14);
  const uint32_t s_free = bar(15);
  const uint32_t p_full = bar(16);
  const uint32_t pv_done = bar(17);
  auto o_full = [&](int b) { return bar(18 + b); };
  auto o_free = [&](int b) { return bar(20 + b); };
  auto l_full = [&](int b) { return bar(22 + b); };
  const uint32_t mma_done = bar(24);

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    for (int i = 0; i < kKStages; ++i) {
      mbar_init(k_full(i), 1);
      mbar_init(k_empty(i), 1);
    }
    for (int i = 0; i < kVStages; ++i) {
      mbar_init(v_full(i), 1);
      mbar_init(v_empty(i), 1);
    }
    mbar_init(s_full, 1);
    mbar_init(s_free, 4);
    for (int b = 0; b < 2; ++b) {
      mbar_init(o_full(b), 1);
      mbar_init(o_free(b), 4);
      mbar_init(l_full(b), 4);
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
    if (elect_one()) tma_prefetch_desc(&tm_qkv);
    __syncwarp();
    // K runs one block ahead of V in issue order: K_{g+1} waits only for an earlier Q K^T,
    // which finishes before the P V that V_g waits for. A tile's Q loads with its first K
    // block, once the previous tile's last Q K^T is done.
    BlockCursor kc, vc;
    kc.init(nqb, n_heads, nseq, blockIdx.x, gridDim.x);
    vc = kc;
    int gk = 0, gv = 0, nq = 0;  // K blocks, V blocks, Q tiles issued
    auto load_k = [&]() {
      if (kc.j == 0) {
        if (kc.i >= 1 &&
            !warp_wait_bounded(q_empty, (kc.i - 1) & 1, abort_flag, err, kDevTimeoutProducer))
          return false;
        if (elect_one()) {
          const int y = kc.seq * P + kc.qb * kBQ;
          mbar_arrive_expect_tx(q_full, kMat);
          tma_load_2d(sQ, &tm_qkv, kc.head * kDh, y, q_full);
          tma_load_2d(sQ + kTile, &tm_qkv, kc.head * kDh + 64, y, q_full);
        }
        __syncwarp();
        ++nq;
      }
      const int st = gk % kKStages;
      if (gk >= kKStages && !warp_wait_bounded(k_empty(st), (gk / kKStages - 1) & 1, abort_flag,
                                               err, kDevTimeoutProducer))
        return false;
      if (elect_one()) {
        const int y = kc.seq * P + kc.j * kBK;
        mbar_arrive_expect_tx(k_full(st), kMat);
        tma_load_2d(sK + st * kMat, &tm_qkv, d + kc.head * kDh, y, k_full(st));
        tma_load_2d(sK + st * kMat + kTile, &tm_qkv, d + kc.head * kDh + 64, y, k_full(st));
      }
      __syncwarp();
      ++gk;
      kc.next();
      return true;
    };
    auto load_v = [&]() {
      const int st = gv % kVStages;
      if (gv >= kVStages && !warp_wait_bounded(v_empty(st), (gv / kVStages - 1) & 1, abort_flag,
                                               err, kDevTimeoutProducer))
        return false;
      if (elect_one()) {
        const int y = vc.seq * P + vc.j * kBK;
        mbar_arrive_expect_tx(v_full(st), kMat);
        tma_load_2d(sV + st * kMat, &tm_qkv, 2 * d + vc.head * kDh, y, v_full(st));
        tma_load_2d(sV + st * kMat + kTile, &tm_qkv, 2 * d + vc.head * kDh + 64, y, v_full(st));
      }
      __syncwarp();
      ++gv;
      vc.next();
      return true;
    };
    // at a tile boundary V_g goes first: the next tile's Q waits for this tile's last Q K^T
    bool ok = kc.valid() ? load_k() : false;
    while (ok && vc.valid()) {
      if (kc.valid() && kc.j != 0) {
        if (!load_k() || !load_v()) break;
      } else {
        if (!load_v() || (kc.valid() && !load_k())) break;
      }
    }
    // copies in flight land before the CTA's shared memory is released
    volatile int no_abort = 0;
    if (nq > 0) warp_wait_bounded(q_full, (nq - 1) & 1, &no_abort, err, kDevTimeoutDrain);
    for (int g = (gk > kKStages ? gk - kKStages : 0); g < gk; ++g)
      warp_wait_bounded(k_full(g % kKStages), (g / kKStages) & 1, &no_abort, err, kDevTimeoutDrain);
    for (int g = (gv > kVStages ? gv - kVStages : 0); g < gv; ++g)
      warp_wait_bounded(v_full(g % kVStages), (g / kVStages) & 1, &no_abort, err, kDevTimeoutDrain);
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    // S_g = Q K_g^T for the next key block is issued before P_g V_g, so it overlaps the
    // softmax of block g. O of a tile accumulates in O[tile & 1].
    BlockCursor sc, pc;
    sc.init(nqb, n_heads, nseq, blockIdx.x, gridDim.x);
    pc = sc;
    int gs = 0, gp = 0;  // S and P V products issued
    auto issue_s = [&]() {
      const int st = gs % kKStages;
      if (sc.j == 0 && !warp_wait_bounded(q_full, sc.i & 1, abort_flag, err, kDevTimeoutMma))
        return false;
      if (!warp_wait_bounded(k_full(st), (gs / kKStages) & 1, abort_flag, err, kDevTimeoutMma))
        return false;
      // the softmax has copied S_{gs-1} to registers
      if (gs >= 1 && !warp_wait_bounded(s_free, (gs - 1) & 1, abort_flag, err, kDevTimeoutMma))
        return false;
      tc_fence_after();
      if (elect_one()) {
        const uint32_t kb = sK + st * kMat;
#pragma unroll
        for (int k = 0; k < kDh / 16; ++k) {
          const uint32_t off = (k >> 2) * kTile + (k & 3) * 32;
          tc_mma_bf16(tmem + kColS, smem_desc_sw128(sQ + off), smem_desc_sw128(kb + off),
                      kIdescQK, k > 0 ? 1u : 0u);
        }
        tc_commit(s_full);
        tc_commit(k_empty(st));
        if (sc.last()) tc_commit(q_empty);
      }
      __syncwarp();
      ++gs;
      sc.next();
      return true;
    };
    auto issue_pv = [&]() {
      const int st = gp % kVStages, ob = pc.i & 1;
      // O[ob] is free once the epilogue has read the tile two back
      if (pc.j == 0 && pc.i >= 2 &&
          !warp_wait_bounded(o_free(ob), ((pc.i - 2) >> 1) & 1, abort_flag, err, kDevTimeoutMma))
        return false;
      if (!warp_wait_bounded(p_full, gp & 1, abort_flag, err, kDevTimeoutMma) ||
          !warp_wait_bounded(v_full(st), (gp / kVStages) & 1, abort_flag, err, kDevTimeoutMma))
        return false;
      tc_fence_after();
      if (elect_one()) {
        const uint32_t vb = sV + st * kMat;
#pragma unroll
        for (int k = 0; k < kBK / 16; ++k) {
          // A: P keys [16k, 16k + 16) from TMEM (8 columns); B: V rows [16k, 16k + 16)
          // (MN-major)
          tc_mma_ts_bf16(tmem + kColO + ob * kDh, tmem + kColP + 8 * k,
                         smem_desc_sw128_mn(vb + k * 2048, kTile), kIdescPV,
                         (pc.j > 0 || k > 0) ? 1u : 0u);
        }
        tc_commit(pv_done);
        tc_commit(v_empty(st));
        if (pc.last()) tc_commit(o_full(ob));
      }
      __syncwarp();
      ++gp;
      pc.next();
      return true;
    };
    // across a tile boundary P V goes first, so that the tile's last block does not wait for
    // the next tile's Q
    bool ok = sc.valid() ? issue_s() : false;
    while (ok && pc.valid()) {
      if (sc.valid() && sc.j != 0) {
        if (!issue_s() || !issue_pv()) break;
      } else {
        if (!issue_pv() || (sc.valid() && !issue_s())) break;
      }
    }
    // every issued MMA has finished before TMEM is released
    if (elect_one()) tc_commit(mma_done);
    __syncwarp();
    volatile int no_abort = 0;
    warp_wait_bounded(mma_done, 0, &no_abort, err, kDevTimeoutDrain);
  } else if (warp < 6) {
    // ---------------------------------------------------------------- softmax (warps 2..5)
    const int q4 = warp & 3;                  // this warp may access TMEM lanes [32 q4, +32)
    const int row = q4 * 32 + lane;           // query row of the tile = TMEM lane
    const uint32_t t_lane = tmem + (static_cast<uint32_t>(q4 * 32) << 16);
    BlockCursor c;
    c.init(nqb, n_heads, nseq, blockIdx.x, gridDim.x);
    float m_ref = -FLT_MAX;                   // reference maximum, log2 domain
    float l = 0.f;                            // row sum of the probabilities
    int g = 0;
    while (c.valid()) {
      const int ob = c.i & 1, j = c.j;
      if (!warp_wait_bounded(s_full, g & 1, abort_flag, err, kDevTimeoutEpilogue)) break;
      tc_fence_after();
      float s[kBK];
      tc_ld_x64(t_lane + kColS, *reinterpret_cast<float(*)[64]>(s));
      tc_ld_x64(t_lane + kColS + 64, *reinterpret_cast<float(*)[64]>(s + 64));
      tc_wait_ld();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(s_free);  // S_g is in registers: Q K_{g+1}^T may overwrite it
      // maximum raw score over the visible keys (on the diagonal block, the tile's last, key
      // c is visible to row `row` iff c <= row), eight chains; the scale (> 0) comes after
      if (c.last()) {
#pragma unroll
        for (int k = 1; k < kBK; ++k)
          if (k > row) s[k] = -INFINITY;
      }
      float pm[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) pm[i] = s[i];
#pragma unroll
      for (int k = 8; k < kBK; ++k) pm[k & 7] = fmaxf(pm[k & 7], s[k]);
      const float mx = fmaxf(fmaxf(fmaxf(pm[0], pm[1]), fmaxf(pm[2], pm[3])),
                             fmaxf(fmaxf(pm[4], pm[5]), fmaxf(pm[6], pm[7]))) *
                       scale_log2;
      bool rescale = false;
      float corr = 1.f;
      if (j == 0) {
        m_ref = mx;
        l = 0.f;
      } else if (mx > m_ref + 8.f) {
        corr = ex2(m_ref - mx);
        m_ref = mx;
        rescale = true;
      }
      // P_g = 2^(scale s - m_ref) in registers (bf16 pairs) before any wait
      float ps[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) ps[i] = 0.f;
      uint32_t w[kBK / 2];
#pragma unroll
      for (int i = 0; i < kBK / 2; ++i) {
        const float p0 = ex2(fmaf(s[2 * i], scale_log2, -m_ref));
        const float p1 = ex2(fmaf(s[2 * i + 1], scale_log2, -m_ref));
        ps[(2 * i) & 7] += p0;
        ps[(2 * i + 1) & 7] += p1;
        w[i] = pack_bf16x2(p0, p1);
      }
      l = l * corr + (((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7])));
      // P_{g-1} V_{g-1} has finished: P in TMEM may be overwritten and O is stable
      if (g > 0 &&
          !warp_wait_bounded(pv_done, (g - 1) & 1, abort_flag, err, kDevTimeoutEpilogue))
        break;
      tc_fence_after();
      if (__any_sync(0xffffffffu, rescale)) {
        const uint32_t t_o = t_lane + kColO + ob * kDh;
#pragma unroll 1
        for (int h = 0; h < 4; ++h) {
          uint32_t o[32];
          tc_ld_32x32b_x32(t_o + 32 * h, o);
          tc_wait_ld();
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * corr);
          tc_st_x32(t_o + 32 * h, o);
        }
        tc_wait_st();
      }
      tc_st_x32(t_lane + kColP, *reinterpret_cast<uint32_t(*)[32]>(w));
      tc_st_x32(t_lane + kColP + 32, *reinterpret_cast<uint32_t(*)[32]>(w + 32));
      tc_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full);
      if (c.last()) {
        // hand the row sum to the epilogue; its copy of the tile two back has been read
        if (c.i >= 2 &&
            !warp_wait_bounded(o_free(ob), ((c.i - 2) >> 1) & 1, abort_flag, err,
                               kDevTimeoutEpilogue))
          break;
        l_sm[ob * kBQ + row] = l;
        __syncwarp();
        if (lane == 0) mbar_arrive(l_full(ob));
      }
      ++g;
      c.next();
    }
  } else {
    // ---------------------------------------------------------------- epilogue (warps 6..9)
    const int q4 = warp & 3;
    const int row = q4 * 32 + lane;
    const uint32_t t_lane = tmem + (static_cast<uint32_t>(q4 * 32) << 16);
    BlockCursor c;
    c.init(nqb, n_heads, nseq, blockIdx.x, gridDim.x);
    for (; c.valid(); c.t += c.stride, ++c.i, c.decode()) {
      const int ob = c.i & 1;
      if (!warp_wait_bounded(o_full(ob), (c.i >> 1) & 1, abort_flag, err, kDevTimeoutEpilogue) ||
          !warp_wait_bounded(l_full(ob), (c.i >> 1) & 1, abort_flag, err, kDevTimeoutEpilogue))
        break;
      tc_fence_after();
      const float inv = 1.f / l_sm[ob * kBQ + row];
      const int q = c.qb * kBQ + row;
      __nv_bfloat16* orow = out + static_cast<size_t>(c.seq * P + q) * ld_out + c.head * kDh;
#pragma unroll 1
      for (int h = 0; h < 4; ++h) {
        uint32_t o[32];
        tc_ld_32x32b_x32(t_lane + kColO + ob * kDh + 32 * h, o);
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
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(o_free(ob));
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
  int dev = 0, nsm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || nsm < 1)
    return -1;
  int* err = device_error_word();
  if (err == nullptr) return -1;
  const int64_t d = n_heads * head_dim;
  CUtensorMap map;
  if (!make_tma_map(&map, qkv, nseq * P, 3 * d, ld, 128, false)) return -2;
  const int64_t ntiles = ((P + kBQ - 1) / kBQ) * n_heads * nseq;
  const unsigned grid = static_cast<unsigned>(ntiles < nsm ? ntiles : nsm);
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(head_dim));
  causal_attention_tc_kernel<<<grid, kThreads, kSmem, st>>>(
      map, static_cast<int>(P), static_cast<int>(d), static_cast<int>(n_heads),
      static_cast<int>(nseq), scale_log2, static_cast<__nv_bfloat16*>(out),
      static_cast<int>(ld_out), err);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace hydra
