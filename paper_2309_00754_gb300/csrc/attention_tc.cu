// Causal self-attention of the Llama decoder on the 5th-generation tensor cores (tcgen05 +
// TMEM + TMA), for both streams at once (each stream's sequences are separate rows):
//     o = softmax(q k^T / sqrt(Dh) + causal mask) v,   head dim Dh = 128
// q, k, v are the column blocks [0, d), [d, 2d), [2d, 3d) of the fused projection output
// (row stride ld); o is written to columns [h Dh, (h + 1) Dh) of out.
//
// Persistent CTAs (one per SM) take units of two adjacent query tiles of 128 rows of one
// (sequence, head), longest first; key/value blocks of 128 rows; flash attention with an
// online softmax. Each K / V block staged in shared memory feeds both tiles, so a block costs
// half the fill traffic per unit of MMA work that one tile per CTA would, and the two tiles
// take turns on the tensor pipe: while one tile's softmax works, the other tile's products run.
//  * warp 0 moves Q_a, Q_b per unit and the K / V blocks through one 3-stage ring with TMA
//    (128-byte swizzle, [128 rows x 64] boxes), in the order the tiles first use them
//    (K_0, V_0, K_1, V_1, ...); the ring runs on across units, and the next unit's first
//    blocks are prefetched into L2 a few blocks before a unit ends (in the longest-first unit
//    order; see UnitCursor). Warp 1 owns TMEM (S_a,
//    S_b, O_a, O_b: 4 x 128 fp32 columns);
//  * warps 4..7 (tile a) and 8..11 (tile b) each run their tile: thread i owns query row i
//    (TMEM lane i), so row maxima and sums need no shuffles, and the group's first warp issues
//    the tile's tcgen05.mma from one elected lane: per key block j, S_x = Q_x K_j^T, then,
//    once the softmax has written P_x as bf16 pairs over the first 64 columns of S_x,
//    O_x += P_x V_j (P_x is the A operand, read from TMEM, so it costs no shared-memory
//    bandwidth) and S_x = Q_x K_{j+1}^T right behind it: the tcgen05.mma operations one
//    thread issues execute in issue order, so the next S, which overwrites the columns of
//    P_x, cannot overtake the P V products that read them. A finished
//    tile is normalised into a staging buffer and stored with TMA (one 128-byte line per row
//    of a box rather than 16-byte pieces of 128 rows), while the tile's next unit runs. The running
//    maximum is a reference value that moves only when a row's maximum grows by more than
//    2^8 (then the thread rescales its O row in TMEM); O and the row sum l share the
//    reference, so O / l is exact either way and every p stays at most 2^8.
// The probabilities enter P V as bf16 (8 mantissa bits, relative error at most 2^-9); the row
// sum l accumulates them in fp32.
#include <float.h>

#include <algorithm>
#include <vector>

#include "common.cuh"
#include "kernels.h"

namespace hydra {
namespace attn_tc {

constexpr int kDh = 128;
constexpr int kBQ = 128;                    // queries per tile (MMA M, TMEM lanes)
constexpr int kBK = 128;                    // keys per block
constexpr int kThreads = 384;               // warpgroup 0: TMA producer (warp 0), TMEM owner
                                            // (warp 1); warpgroups 1, 2: tiles a, b
// Registers per thread after setmaxnreg: 384 threads x 168 at launch = 128 x 56 + 256 x 224
constexpr uint32_t kRegsLight = 56;
constexpr uint32_t kRegsTile = 224;
static_assert(128 * kRegsLight + 256 * kRegsTile <= kThreads * 168, "register split");
constexpr int kTile = 128 * 64 * 2;         // [128 rows x 64 bf16] swizzled tile: 16 KiB
constexpr int kMat = 2 * kTile;             // [128 x 128] bf16 operand: 32 KiB
constexpr int kOffQ = 0;                    // Q_a, Q_b
constexpr int kStages = 3;                  // one ring for K and V blocks: K_0, V_0, K_1, ...
constexpr int kOffKV = kOffQ + 2 * kMat;
constexpr int kOffOut = kOffKV + kStages * kMat;  // output staging: one tile per tile
constexpr int kOffBar = kOffOut + 2 * kMat;
constexpr int kNumBars = 4 + 2 * kStages + 4;
constexpr int kSmem = 1024 + kOffBar + kNumBars * 8 + 16;
static_assert(kSmem <= 232448, "shared memory per CTA");
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS = 0;               // S_a, S_b: 128 fp32 columns each; P_x (bf16
                                            // pairs) overwrites the first 64 columns of S_x
constexpr uint32_t kColO = 256;             // O_a, O_b: 128 fp32 columns each

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

// Bring the box at (x, y) of a tensor map into L2 (no shared-memory destination).
__device__ __forceinline__ void tma_prefetch_l2_2d(const CUtensorMap* map, int x, int y) {
  asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y)
               : "memory");
}

// Store the box at (x, y, z) of a 3-D tensor map from shared memory at src (TMA; elements
// outside the tensor are not written).
__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, uint32_t src, int x, int y,
                                             int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%1, %2, %3}], [%4];" ::"l"(
          reinterpret_cast<uint64_t>(map)),
      "r"(x), "r"(y), "r"(z), "r"(src)
      : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// the shared-memory source of every committed bulk store has been read
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
// every committed bulk store has completed
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// barrier over the 128 threads of one warpgroup (named barrier id 1 + x)
__device__ __forceinline__ void wg_sync(int x) {
  asm volatile("bar.sync %0, 128;" ::"r"(1 + x) : "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c,
                                             uint32_t e) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c),
               "r"(e)
               : "memory");
}

// Packed fp32 pairs (sm_100 and later execute add / fma on two fp32 lanes per instruction)
// and a three-input maximum, for the softmax's elementwise steps. (Moving part of the
// exponentials to the FMA pipe with a cubic was measured slower at every fraction tried.)
__device__ __forceinline__ uint64_t f2_pack(float a, float b) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
  return r;
}
__device__ __forceinline__ void f2_unpack(uint64_t v, float& a, float& b) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ float max3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
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


// This CTA's work: units t = blockIdx.x + i * gridDim.x (i = 0, 1, ...). Unit (p, head, seq)
// holds the two query tiles qa = 2p and qb = 2p + 1 (qb only when it exists): tile a runs key
// blocks 0..qa, tile b 0..qb, and every key block the two share is loaded once for both. Two
// orders of the units t:
//  * longest first: t -> (p, head, seq) with the largest p (most key blocks) first;
//  * grouped: the units of one (head, sequence) consecutive, longest first within it, so
//    that they run at the same time on neighbouring CTAs and read the key / value blocks
//    they share from DRAM once (the longest-first order runs them waves apart, when the
//    blocks have left L2).
// The launcher takes the grouped order unless it raises the busiest CTA's load (in key
// blocks) of the static round-robin assignment by more than 5 % over the longest-first order.
struct UnitCursor {
  int t;               // unit
  int p, head, seq;    // decoded unit
  int na, nb, nblk;    // key blocks of tile a, of tile b (0: no tile b), of the unit
  // the loop-invariant sizes are recomputed from the kernel arguments (constant bank) rather
  // than kept in registers: the producer and MMA warps run with few registers
  __host__ __device__ static int units(int P, int heads, int nseq) {
    return (((P + kBQ - 1) / kBQ + 1) / 2) * heads * nseq;
  }
  __host__ __device__ void decode(int P, int heads, int nseq, int grouped) {
    const int nqb = (P + kBQ - 1) / kBQ;
    const int npairs = (nqb + 1) / 2;
    if (grouped) {
      const int g = t / npairs;
      p = npairs - 1 - t % npairs;
      head = g % heads;
      seq = g / heads;
    } else {
      const int hs = heads * nseq;
      p = npairs - 1 - t / hs;
      const int r = t % hs;
      head = r % heads;
      seq = r / heads;
    }
    na = 2 * p + 1;
    nb = (2 * p + 1 < nqb) ? 2 * p + 2 : 0;
    nblk = nb > 0 ? nb : na;
  }
};

__global__ void __launch_bounds__(kThreads, 1)
    causal_attention_tc_kernel(const __grid_constant__ CUtensorMap tm_qkv,
                               const __grid_constant__ CUtensorMap tm_out, int P, int d,
                               int n_heads, int nseq, int grouped, float scale_log2, int* err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kOffBar);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + kNumBars);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int nunits = UnitCursor::units(P, n_heads, nseq);

  const uint32_t sbase = smem_u32(smem);
  auto sQ = [&](int x) { return sbase + kOffQ + x * kMat; };
  auto sKV = [&](int st) { return sbase + kOffKV + st * kMat; };
  auto bar = [&](int i) { return smem_u32(&bars[i]); };
  auto q_full = [&](int x) { return bar(0 + x); };
  auto q_empty = [&](int x) { return bar(2 + x); };
  auto kv_full = [&](int st) { return bar(4 + st); };
  auto kv_empty = [&](int st) { return bar(4 + kStages + st); };
  auto s_full = [&](int x) { return bar(4 + 2 * kStages + x); };
  auto pv_done = [&](int x) { return bar(6 + 2 * kStages + x); };

  if (threadIdx.x == 0) {
    for (int x = 0; x < 2; ++x) {
      mbar_init(q_full(x), 1);
      mbar_init(q_empty(x), 1);
      mbar_init(s_full(x), 1);
      mbar_init(pv_done(x), 1);
    }
    // a K or V block is released by each of the two tiles (a block only one tile uses is
    // released twice by that tile)
    for (int i = 0; i < kStages; ++i) {
      mbar_init(kv_full(i), 1);
      mbar_init(kv_empty(i), 2);
    }
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

  if (warp < 4) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegsLight));
    if (warp == 0) {
      // -------------------------------------------------------------- TMA producer
      // Per unit: Q_a, K_0, Q_b, V_0, K_1, V_1, ..., the order in which the tiles first need
      // them; the ring runs on across units
      if (elect_one()) {
        tma_prefetch_desc(&tm_qkv);
        tma_prefetch_desc(&tm_out);
      }
      __syncwarp();
      UnitCursor c = {};
      int pos = 0, nq[2] = {0, 0};  // ring positions filled, Q tiles loaded per tile
      bool ok = true;
      auto load_q = [&](int x) {
        if (nq[x] >= 1 && !warp_wait_bounded(q_empty(x), (nq[x] - 1) & 1, abort_flag, err,
                                             kDevTimeoutProducer))
          return false;
        if (elect_one()) {
          const int y = c.seq * P + (2 * c.p + x) * kBQ;
          mbar_arrive_expect_tx(q_full(x), kMat);
          tma_load_2d(sQ(x), &tm_qkv, c.head * kDh, y, q_full(x));
          tma_load_2d(sQ(x) + kTile, &tm_qkv, c.head * kDh + 64, y, q_full(x));
        }
        __syncwarp();
        ++nq[x];
        return true;
      };
      // K (kv = 1) or V (kv = 2) of key block j
      auto load_kv = [&](int kv, int j) {
        const int st = pos % kStages;
        if (pos >= kStages && !warp_wait_bounded(kv_empty(st), (pos / kStages - 1) & 1,
                                                 abort_flag, err, kDevTimeoutProducer))
          return false;
        if (elect_one()) {
          const int y = c.seq * P + j * kBK;
          const int x0 = kv * d + c.head * kDh;
          mbar_arrive_expect_tx(kv_full(st), kMat);
          tma_load_2d(sKV(st), &tm_qkv, x0, y, kv_full(st));
          tma_load_2d(sKV(st) + kTile, &tm_qkv, x0 + 64, y, kv_full(st));
        }
        __syncwarp();
        ++pos;
        return true;
      };
      // L2 prefetch of the next unit's Q tiles and first two K / V blocks, a few blocks before
      // this unit ends: every CTA reaches a unit boundary at about the same time, and the
      // loads there would otherwise queue behind each other in DRAM
      auto prefetch_next = [&]() {
        UnitCursor nx;
        nx.t = c.t + gridDim.x;
        if (nx.t >= nunits || !elect_one()) return;
        nx.decode(P, n_heads, nseq, grouped);
        const int y0 = nx.seq * P;
        for (int x = 0; x < (nx.nb > 0 ? 2 : 1); ++x)
          for (int h = 0; h < 2; ++h)
            tma_prefetch_l2_2d(&tm_qkv, nx.head * kDh + 64 * h, y0 + (2 * nx.p + x) * kBQ);
        for (int j = 0; j < (nx.nblk < 2 ? nx.nblk : 2); ++j)
          for (int kv = 1; kv <= 2; ++kv)
            for (int h = 0; h < 2; ++h)
              tma_prefetch_l2_2d(&tm_qkv, kv * d + nx.head * kDh + 64 * h, y0 + j * kBK);
      };
      for (c.t = blockIdx.x; ok && c.t < nunits; c.t += gridDim.x) {
        c.decode(P, n_heads, nseq, grouped);
        // prefetch after this block's loads (longest-first order only: with the grouped
        // order the next unit's blocks are mostly in L2 already, and the prefetch measured slower)
        const int jpf = grouped ? -1 : (c.nblk > 3 ? c.nblk - 3 : 0);
        ok = load_q(0) && load_kv(1, 0);
        if (ok && c.nb > 0) ok = load_q(1);
        if (ok) ok = load_kv(2, 0);
        if (ok && jpf == 0) prefetch_next();
        __syncwarp();
        for (int j = 1; ok && j < c.nblk; ++j) {
          ok = load_kv(1, j) && load_kv(2, j);
          if (ok && j == jpf) prefetch_next();
          __syncwarp();
        }
      }
      // copies in flight land before the CTA's shared memory is released
      volatile int no_abort = 0;
      for (int x = 0; x < 2; ++x)
        if (nq[x] > 0)
          warp_wait_bounded(q_full(x), (nq[x] - 1) & 1, &no_abort, err, kDevTimeoutDrain);
      for (int g = (pos > kStages ? pos - kStages : 0); g < pos; ++g)
        warp_wait_bounded(kv_full(g % kStages), (g / kStages) & 1, &no_abort, err,
                          kDevTimeoutDrain);
    }
  } else {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kRegsTile));
    // -------------------------------------------------------------- tiles (warps 4..11)
    // Warps 4..7 own tile a, warps 8..11 tile b; thread i of a group owns query row i (TMEM
    // lane i). Each group runs its tile's softmax and issues the tile's products itself:
    // once P_x is in TMEM, one of its warps issues P_x V_j and then Q_x K_{j+1}^T (in issue
    // order behind the P V products that read P_x, which the next S overwrites), so no other
    // warp sits on
    // the path from a finished P to the tensor pipe. The two groups' products interleave on
    // the pipe: one tile's softmax overlaps the other tile's products.
    const int x = warp < 8 ? 0 : 1;
    const int q4 = warp & 3;                  // this warp may access TMEM lanes [32 q4, +32)
    const int row = q4 * 32 + lane;           // query row of the tile = TMEM lane
    // the warp that issues the tile's products: sub-partition 1 for tile a, 2 for tile b, so
    // that neither shares a scheduler with the other issuer or with the TMA producer (warp 0)
    const bool issuer = (q4 == 1 + x);
    const uint32_t t_lane = tmem + (static_cast<uint32_t>(q4 * 32) << 16);
    const uint32_t t_s = t_lane + kColS + x * 128;
    const uint32_t t_o = t_lane + kColO + x * kDh;
    const uint32_t s_stage = sbase + kOffOut + x * kMat;  // this tile's output staging
    int gs = 0, nqu = 0;                      // S consumed, units begun (Q tiles)
    int kbase = 0;                            // ring block index of the unit's key block 0
    bool s0_issued = false;                   // this unit's first Q K^T was issued already
    bool ok = true;
    // Q_x K^T of the block at ring position kpos (issuer warp); rel: releases of its stage
    auto issue_s = [&](bool first, int kpos, int rel, bool last_s) {
      if (first && !warp_wait_bounded(q_full(x), nqu & 1, abort_flag, err, kDevTimeoutMma))
        return false;
      const int st = kpos % kStages;
      if (!warp_wait_bounded(kv_full(st), (kpos / kStages) & 1, abort_flag, err, kDevTimeoutMma))
        return false;
      tc_fence_after();
      if (elect_one()) {
        // descriptors of the tile bases; a k-step adds its byte offset / 16 to the address
        // field (every shared address here is below 2^18, so the field cannot carry over)
        const uint64_t dq = smem_desc_sw128(sQ(x));
        const uint64_t dk = smem_desc_sw128(sKV(st));
#pragma unroll
        for (int k = 0; k < kDh / 16; ++k) {
          const uint32_t off = ((k >> 2) * kTile + (k & 3) * 32) >> 4;
          tc_mma_bf16(tmem + kColS + x * 128, dq + off, dk + off, kIdescQK, k > 0 ? 1u : 0u);
        }
        tc_commit(s_full(x));
        for (int i = 0; i < rel; ++i) tc_commit(kv_empty(st));
        if (last_s) tc_commit(q_empty(x));
      }
      __syncwarp();
      if (first) ++nqu;
      return true;
    };
    // P_x V of the block at ring position vpos (issuer warp)
    auto issue_pv = [&](bool first, int vpos, int rel) {
      const int st = vpos % kStages;
      if (!warp_wait_bounded(kv_full(st), (vpos / kStages) & 1, abort_flag, err, kDevTimeoutMma))
        return false;
      tc_fence_after();
      if (elect_one()) {
        const uint64_t dv = smem_desc_sw128_mn(sKV(st), kTile);
#pragma unroll
        for (int k = 0; k < kBK / 16; ++k)
          tc_mma_ts_bf16(tmem + kColO + x * kDh, tmem + kColS + x * 128 + 8 * k,
                         dv + ((k * 2048) >> 4), kIdescPV, (!first || k > 0) ? 1u : 0u);
        tc_commit(pv_done(x));
        for (int i = 0; i < rel; ++i) tc_commit(kv_empty(st));
      }
      __syncwarp();
      return true;
    };
    float m_ref = -FLT_MAX;                   // reference maximum, log2 domain
    float l = 0.f;                            // row sum of the probabilities
    UnitCursor c;
    for (c.t = blockIdx.x; ok && c.t < nunits; c.t += gridDim.x) {
      c.decode(P, n_heads, nseq, grouped);
      const int n = x == 0 ? c.na : c.nb;     // this tile's key blocks (0: no tile b)
      const int on = x == 0 ? c.nb : c.na;    // the other tile's
      const int J = c.nblk;
      if (n == 0) {
        kbase += J;
        s0_issued = false;
        continue;
      }
      // ring positions: K_j at 2 (kbase + j), V_j right after it
      if (!s0_issued && issuer) ok = issue_s(true, 2 * kbase, on > 0 ? 1 : 2, n == 1);
      for (int j = 0; ok && j < n; ++j) {
        if (!warp_wait_bounded(s_full(x), gs & 1, abort_flag, err, kDevTimeoutEpilogue)) {
          ok = false;
          break;
        }
        ++gs;
        tc_fence_after();
        float sv[kBK];
        tc_ld_x64(t_s, *reinterpret_cast<float(*)[64]>(sv));
        tc_ld_x64(t_s + 64, *reinterpret_cast<float(*)[64]>(sv + 64));
        tc_wait_ld();
        // the diagonal block (the tile's last): key c is visible to row `row` iff c <= row
        const bool diag = (j == n - 1);
        if (diag) {
#pragma unroll
          for (int k = 1; k < kBK; ++k)
            if (k > row) sv[k] = -INFINITY;
        }
        float pm[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) pm[i] = -FLT_MAX;
#pragma unroll
        for (int i = 0; i < kBK / 2; ++i) pm[i & 7] = max3(pm[i & 7], sv[2 * i], sv[2 * i + 1]);
        const float mx = max3(max3(pm[0], pm[1], pm[2]), max3(pm[3], pm[4], pm[5]),
                              fmaxf(pm[6], pm[7])) *
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
        // P = 2^(scale s - m_ref) as bf16 pairs over the first 64 columns of S_x; the argument
        // and the row sum in packed pairs
        const uint64_t sc2 = f2_pack(scale_log2, scale_log2), nm2 = f2_pack(-m_ref, -m_ref);
        uint64_t acc[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[i] = f2_pack(0.f, 0.f);
        uint32_t w[kBK / 2];
#pragma unroll
        for (int i = 0; i < kBK / 2; ++i) {
          float a0, a1;
          f2_unpack(f2_fma(f2_pack(sv[2 * i], sv[2 * i + 1]), sc2, nm2), a0, a1);
          const float p0 = ex2(a0), p1 = ex2(a1);
          acc[i & 3] = f2_add(acc[i & 3], f2_pack(p0, p1));
          w[i] = pack_bf16x2(p0, p1);
        }
        float ps[8];
#pragma unroll
        for (int i = 0; i < 4; ++i) f2_unpack(acc[i], ps[2 * i], ps[2 * i + 1]);
        l = l * corr + (((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7])));
        // O_x holds the sum through the previous block (that P V finished before this S was
        // issued): rescale the row when the reference moved
        if (__any_sync(0xffffffffu, rescale)) {
#pragma unroll 1
          for (int h = 0; h < 4; ++h) {
            uint32_t o[32];
            tc_ld_32x32b_x32(t_o + 32 * h, o);
            tc_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * corr);
            tc_st_x32(t_o + 32 * h, o);
            tc_wait_st();
          }
        }
        tc_st_x32(t_s, *reinterpret_cast<uint32_t(*)[32]>(w));
        tc_st_x32(t_s + 32, *reinterpret_cast<uint32_t(*)[32]>(w + 32));
        tc_wait_st();
        tc_fence_before();
        wg_sync(x);  // P_x of the whole tile is in TMEM
        if (issuer) {
          ok = issue_pv(j == 0, 2 * (kbase + j) + 1, j < on ? 1 : 2);
          if (ok && j + 1 < n) {
            ok = issue_s(false, 2 * (kbase + j + 1), j + 1 < on ? 1 : 2, j + 1 == n - 1);
          } else if (ok) {
            // the next unit's first Q_x K^T, if it has tile x: its stage meanwhile fills
            UnitCursor nx;
            nx.t = c.t + gridDim.x;
            s0_issued = false;
            if (nx.t < nunits) {
              nx.decode(P, n_heads, nseq, grouped);
              const int nn = x == 0 ? nx.na : nx.nb, non = x == 0 ? nx.nb : nx.na;
              if (nn > 0) {
                ok = issue_s(true, 2 * (kbase + J), non > 0 ? 1 : 2, nn == 1);
                s0_issued = true;
              }
            }
          }
        }
      }
      if (!ok) break;
      // the finished tile (its last P V, the gs-th, is done; the parity wait cannot alias an
      // older phase: the tile's last S completed after every earlier product of the issuing
      // thread, so only this P V can be outstanding): O_x / l as bf16 rows, staged in
      // shared memory as two 128-byte-swizzled TMA boxes of 64 columns and stored with TMA;
      // the staging buffer is reused only once the stores of the previous unit have read it
      if (issuer) {
        if (elect_one()) bulk_wait_read();
        __syncwarp();
      }
      if (!warp_wait_bounded(pv_done(x), (gs - 1) & 1, abort_flag, err, kDevTimeoutEpilogue)) {
        ok = false;
        break;
      }
      tc_fence_after();
      {
        uint32_t o[4][32];
#pragma unroll
        for (int q = 0; q < 4; ++q) tc_ld_32x32b_x32(t_o + 32 * q, o[q]);
        tc_wait_ld();
        const float inv = 1.f / l;
        wg_sync(x);  // the previous unit's stores have read the staging buffer
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const uint32_t box = s_stage + (q >> 1) * kTile + row * 128;
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            auto f = [&](int e) { return __uint_as_float(o[q][8 * i + e]) * inv; };
            const int chunk = 4 * (q & 1) + i;
            st_shared_v4(box + ((chunk ^ (row & 7)) << 4), pack_bf16x2(f(0), f(1)),
                         pack_bf16x2(f(2), f(3)), pack_bf16x2(f(4), f(5)), pack_bf16x2(f(6), f(7)));
          }
        }
      }
      fence_proxy_async_smem();
      wg_sync(x);
      if (issuer) {
        if (elect_one()) {
          for (int h = 0; h < 2; ++h)
            tma_store_3d(&tm_out, s_stage + h * kTile, c.head * kDh + 64 * h, (2 * c.p + x) * kBQ,
                         c.seq);
          bulk_commit();
        }
        __syncwarp();
      }
      kbase += J;
    }
    if (issuer && elect_one()) bulk_wait_all();
    __syncwarp();
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
  CUtensorMap map, map_out;
  if (!make_tma_map(&map, qkv, nseq * P, 3 * d, ld, 128, false)) return -2;
  // output as nseq planes of [P, d]: a tile's rows past its sequence are not stored
  if (!make_tma_map_3d(&map_out, out, d, P, nseq, ld_out, P * ld_out, kBQ)) return -2;
  const int64_t nunits = ((P + 2 * kBQ - 1) / (2 * kBQ)) * n_heads * nseq;
  const unsigned grid = static_cast<unsigned>(nunits < nsm ? nunits : nsm);
  // unit order: grouped unless it loads the busiest CTA of the static round-robin assignment
  // with more than 5 % more key blocks than the longest-first order does (its shared reads
  // measured worth that much: 8 x 768 x 32 heads, equal loads, 64 -> 58 us; 16 x 768 x 32
  // heads, 46 against 44 blocks, 119 -> 102 us; 16 x 300 x 12 heads, 9 against 8, slower).
  // The choice for the last shape is kept.
  struct OrderChoice {
    int64_t nseq, P, heads;
    unsigned grid;
    int grouped;
  };
  static thread_local OrderChoice last = {-1, -1, -1, 0, 0};
  if (last.nseq != nseq || last.P != P || last.heads != n_heads || last.grid != grid) {
    auto busiest = [&](int grouped) {
      std::vector<int64_t> load(grid, 0);
      UnitCursor c;
      for (int64_t t = 0; t < nunits; ++t) {
        c.t = static_cast<int>(t);
        c.decode(static_cast<int>(P), static_cast<int>(n_heads), static_cast<int>(nseq), grouped);
        load[t % grid] += c.nblk;
      }
      return *std::max_element(load.begin(), load.end());
    };
    last = {nseq, P, n_heads, grid, busiest(1) * 20 <= busiest(0) * 21 ? 1 : 0};
  }
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(head_dim));
  causal_attention_tc_kernel<<<grid, kThreads, kSmem, st>>>(
      map, map_out, static_cast<int>(P), static_cast<int>(d), static_cast<int>(n_heads),
      static_cast<int>(nseq), last.grouped, scale_log2, err);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace hydra
