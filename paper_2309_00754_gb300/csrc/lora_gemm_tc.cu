// Dual-output LoRA linear on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
// One frozen weight W serves both roles of the Hydra model (§3 Dynamic LoRA: the
// reference policy is the actor with its LoRA parameters ignored):
//     y_off = x_off W^T                             (LoRA off: reference / reward stream)
//     y_on  = x_on  W^T + u B^T,  u = s x_on A^T    (LoRA on: actor / critic stream)
// Storage: x [M, K], W [N, K], u [M, r], B [N, r], all bf16 row-major (K-major operands).
//
// Persistent kernel, one CTA per SM, tiles of 128 x 256 (k-step 64) taken round-robin.
// Warp 0 issues TMA loads into a 4-stage shared-memory ring, warp 1 owns TMEM and issues
// tcgen05.mma from one thread, warps 2..5 drain TMEM (warp w reads lanes 32*(w%4)..+31)
// and store through swizzled shared memory with TMA. TMEM holds two 128 x 256 fp32
// accumulators, so the epilogue of one tile overlaps the main loop of the next.
//
// Two tile kinds:
//  * shared input (x_on == x_off) with LoRA: the tile's x W^T is drained to y_off; the
//    LoRA k-block(s) (u B^T) then accumulate on top of the same accumulator and the
//    epilogue drains y_on. The LoRA k-blocks of tile j are placed in the ring a few
//    k-blocks into tile j+1, so the y_off drain overlaps tensor-core work. One read of
//    each W tile yields both outputs.
//  * stacked streams (x_on != x_off): tiles of the off stream produce y_off; tiles of the
//    on stream run the main loop followed directly by the LoRA k-blocks
//    ([x_on | u] [W | B]^T) and produce y_on. Off and on tiles of one (m, n) block are
//    adjacent in the schedule, so each W tile comes from HBM once and again from L2.
#include <float.h>

#include "common.cuh"
#include "kernels.h"

namespace hydra {
namespace tcgemm {

constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 64;
constexpr int STAGES = 4;
constexpr int A_TILE = BM * BK * 2;  // 16 KiB
constexpr int B_TILE = BN * BK * 2;  // 32 KiB
constexpr int STAGE_BYTES = A_TILE + B_TILE;
constexpr int NUM_THREADS = 192;
constexpr int EPI_WARPS = 4;
constexpr int STAGING_BYTES = 32 * 128;  // 32 rows x 128 B per epilogue-warp buffer
constexpr uint32_t TMEM_COLS = 512;      // two accumulators of 256 fp32 columns
constexpr int DEFER = 8;                 // LoRA k-blocks of tile j follow k-block DEFER-1 of tile j+1
constexpr int NUM_BARS = 2 * STAGES + 7;
constexpr int SMEM_BYTES =
    1024 + STAGES * STAGE_BYTES + EPI_WARPS * 2 * STAGING_BYTES + NUM_BARS * 8 + 16;
constexpr uint32_t IDESC = idesc_bf16_f32(BM, BN);

// Epilogue modes (what a drained accumulator tile becomes):
//  EPI_STORE    y = acc (bf16 or fp32)
//  EPI_SWIGLU   columns [0, 128) of the tile are gate, [128, 256) up for the same 128
//               features: y[:, n0/2 + j] = bf16(silu(bf16(gate_j)) * bf16(up_j))
//  EPI_RESIDUAL y (fp32 residual stream) += float(bf16(acc)) by TMA reduce-add in L2
//  EPI_ROPE     y = bf16 rotary embedding of bf16(acc) on columns [0, rope_cols) (heads of
//               128, rotate-half pairs (i, i + 64), position row % rope_P), bf16(acc) after
//  EPI_LOGSOFTMAX  nothing stored per column: per (row, 256-column tile) the fp32 logits'
//               (max, sum exp(z - max)) go to a partials array [rows][n_tiles] (float2), and
//               the logit of the row's sampled token to targets [rows] if it is in the tile
enum { EPI_STORE = 0, EPI_SWIGLU = 1, EPI_RESIDUAL = 2, EPI_ROPE = 3, EPI_LOGSOFTMAX = 4 };

struct Params {
  int M, N, K;
  int epi;
  int kb_main;  // ceil(K / BK)
  int kb_lora;  // ceil(r / BK); 0 = no LoRA
  int r;
  int shared_x;   // 1 = x_on is x_off
  int deferred;   // shared input with LoRA and both outputs: y_off drain, then LoRA
  int streams;    // 1 (shared) or 2 (stacked)
  int m_tiles, n_tiles, total_tiles;
  int m_group;  // CTA-pair kernel: 0 = m fastest over all of M; else groups of m_group
                // m-tiles, m fastest inside a group, then n, then the next group
  int has_off, has_on, has_crit;
  int out_f32;
  int bn;          // tile width in output columns (multiple of 16; 256 for the single-CTA kernel)
  int rope_P, rope_cols;
  const float2* rope_table;  // (cos, sin) [rope_P][64]
  // EPI_LOGSOFTMAX: y_off_ptr / y_on_ptr are the two streams' partials [M][n_tiles]; the
  // streams' targets are lsm_target [2][M]; the token of row m is
  // lsm_ids[(m / lsm_L) * lsm_ids_ld + lsm_ids_off + m % lsm_L]
  float* lsm_target;
  const int32_t* lsm_ids;
  int lsm_L, lsm_ids_ld, lsm_ids_off;
  void* y_off_ptr;  // the outputs as plain pointers, for columns past the last full store chunk
  void* y_on_ptr;
  void* y_crit_ptr;
  int* err;
};

// The kernel's TMA descriptors: inputs of the off, on (actor) and critic streams, W, the
// LoRA operands (u, B) of the on and critic streams, and the three streams' outputs.
struct Maps {
  CUtensorMap x[3];
  CUtensorMap w;
  CUtensorMap u[2];
  CUtensorMap b[2];
  CUtensorMap y[3];
};

struct Tile {
  int stream, m0, n0, n_lora;
};

__device__ __forceinline__ Tile decode(const Params& p, int t) {
  Tile tl;
  tl.stream = t % p.streams;
  t /= p.streams;
  tl.m0 = (t % p.m_tiles) * BM;
  tl.n0 = (t / p.m_tiles) * p.bn;
  // stream 0 is LoRA-off; stream 1 carries the on (actor) LoRA set, stream 2 the critic set
  const bool lora = p.shared_x ? true : (tl.stream >= 1);
  const bool wanted = tl.stream == 2 ? p.has_crit : p.has_on;
  tl.n_lora = (p.kb_lora > 0 && lora && wanted) ? p.kb_lora : 0;
  return tl;
}

__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, uint32_t src, int x, int y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(src)
               : "memory");
}
__device__ __forceinline__ void tma_reduce_add_2d(const CUtensorMap* map, uint32_t src, int x,
                                                  int y) {
  asm volatile(
      "cp.reduce.async.bulk.tensor.2d.global.shared::cta.add.tile.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
          reinterpret_cast<uint64_t>(map)),
      "r"(x), "r"(y), "r"(src)
      : "memory");
}
__device__ __forceinline__ float bf16_round(float v) {
  return __bfloat162float(__float2bfloat16_rn(v));
}
__device__ __forceinline__ void bulk_commit() {
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_read1() {
  asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_all() {
  asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_all_read() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c,
                                             uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c),
               "r"(d)
               : "memory");
}

// Rotary epilogue of one warp's 32 rows (thread `lane` owns row y + lane), one head of 128
// columns at a time: the head's two halves x1 = [0, 64) and x2 = [64, 128) become
// x1 cos - x2 sin and x1 sin + x2 cos with (cos, sin) of pair i at position pos from the
// rotation table, on the bf16-rounded accumulator, each rounding explicit (the rotary kernel
// runs the same operations on the same angles). Both halves are staged (one buffer each)
// and stored as [32 x 64] boxes.
__device__ __forceinline__ void drain_rope(uint32_t lane_taddr, int lane, uint32_t staging,
                                           const Params& p, int y, int n0, const CUtensorMap* t0,
                                           const CUtensorMap* t1) {
  const int row = y + lane;
  const float4* trow = reinterpret_cast<const float4*>(p.rope_table + (row % p.rope_P) * 64);
  for (int h = 0; h < p.bn / 128; ++h) {
    const int col0 = n0 + 128 * h;
    const bool rot = col0 < p.rope_cols;
    if (lane == 0) bulk_wait_all_read();  // both staging buffers are free
    __syncwarp();
#pragma unroll 1
    for (int g = 0; g < 2; ++g) {
      uint32_t x1[32], x2[32];
      tc_ld_32x32b_x32(lane_taddr + 128 * h + 32 * g, x1);
      tc_ld_32x32b_x32(lane_taddr + 128 * h + 64 + 32 * g, x2);
      tc_wait_ld();
      uint32_t o1[16], o2[16];
#pragma unroll
      for (int e = 0; e < 16; ++e) {
        const float a0 = bf16_round(__uint_as_float(x1[2 * e]));
        const float a1 = bf16_round(__uint_as_float(x1[2 * e + 1]));
        const float b0 = bf16_round(__uint_as_float(x2[2 * e]));
        const float b1 = bf16_round(__uint_as_float(x2[2 * e + 1]));
        if (rot) {
          const float4 cs = __ldg(trow + 16 * g + e);  // (cos, sin) of pairs 32 g + 2 e, + 1
          const float c0 = cs.x, s0 = cs.y, c1 = cs.z, s1 = cs.w;
          o1[e] = pack_bf16x2(__fsub_rn(__fmul_rn(a0, c0), __fmul_rn(b0, s0)),
                              __fsub_rn(__fmul_rn(a1, c1), __fmul_rn(b1, s1)));
          o2[e] = pack_bf16x2(__fadd_rn(__fmul_rn(a0, s0), __fmul_rn(b0, c0)),
                              __fadd_rn(__fmul_rn(a1, s1), __fmul_rn(b1, c1)));
        } else {
          o1[e] = pack_bf16x2(a0, a1);
          o2[e] = pack_bf16x2(b0, b1);
        }
      }
      // half rows of the two [32 x 128 B] staging buffers (128-byte swizzle)
      const uint32_t r1 = staging + lane * 128, r2 = staging + STAGING_BYTES + lane * 128;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int u = 4 * g + j;
        st_shared_v4(r1 + ((u ^ (lane & 7)) << 4), o1[4 * j], o1[4 * j + 1], o1[4 * j + 2], o1[4 * j + 3]);
        st_shared_v4(r2 + ((u ^ (lane & 7)) << 4), o2[4 * j], o2[4 * j + 1], o2[4 * j + 2], o2[4 * j + 3]);
      }
    }
    fence_async_smem();
    __syncwarp();
    if (lane == 0) {
      if (y < p.M) {
        for (int half = 0; half < 2; ++half) {
          const int x = col0 + 64 * half;
          if (x >= p.N) continue;
          const uint32_t buf = staging + half * STAGING_BYTES;
          if (t0) tma_store_2d(t0, buf, x, y);
          if (t1) tma_store_2d(t1, buf, x, y);
        }
      }
      bulk_commit();
    }
  }
}

// Log-softmax epilogue of one warp's 32 rows (thread `lane` owns row y + lane): the row's
// fp32 logits in this tile, [n0, n0 + bn) clipped at N, reduce to an online (max, sum of
// exp) pair (the normaliser of Milakov & Gimelshein, as the log-probability kernel keeps
// it) written to partials[row][n0 / bn] of each requested stream; the logit of the row's
// token goes to that stream's target if the token falls in the tile. part0 / part1 are the
// streams' partial arrays (NULL: not requested).
__device__ __forceinline__ void drain_logsoftmax(uint32_t lane_taddr, int lane, const Params& p,
                                                 int y, int n0, void* part0, void* part1) {
  const int row = y + lane;
  const bool live = row < p.M;
  int id = -1;
  if (live) {
    const int s = row / p.lsm_L, t = row - s * p.lsm_L;
    id = p.lsm_ids[static_cast<int64_t>(s) * p.lsm_ids_ld + p.lsm_ids_off + t];
  }
  float m = -FLT_MAX, sum = 0.f, z = 0.f;
  bool hit = false;
  for (int c = 0; c < p.bn / 32; ++c) {
    uint32_t v[32];
    tc_ld_32x32b_x32(lane_taddr + 32 * c, v);
    tc_wait_ld();
    const int col0 = n0 + 32 * c;
    if (col0 >= p.N) break;  // uniform over the warp
    const int nv = min(32, p.N - col0);
    float mx = -FLT_MAX;
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (j < nv) mx = fmaxf(mx, __uint_as_float(v[j]));
    if (mx > m) {
      sum *= __expf(m - mx);
      m = mx;
    }
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (j < nv) sum += __expf(__uint_as_float(v[j]) - m);
    if (id >= col0 && id < col0 + nv) {
      // arithmetic select (exact: every other term is +0), so v stays in registers
      const int k = id - col0;
      float acc = 0.f;
#pragma unroll
      for (int j = 0; j < 32; ++j) acc += (k == j) ? __uint_as_float(v[j]) : 0.f;
      z = acc;
      hit = true;
    }
  }
  if (!live) return;
  const int64_t slot = static_cast<int64_t>(row) * p.n_tiles + n0 / p.bn;
  for (int o = 0; o < 2; ++o) {
    float2* part = static_cast<float2*>(o == 0 ? part0 : part1);
    if (part == nullptr) continue;
    part[slot] = make_float2(m, sum);
    if (hit) p.lsm_target[(part == p.y_on_ptr ? p.M : 0) + row] = z;
  }
}

// Epilogue warp: drain the warp's 32 accumulator rows (TMEM lanes) of one tile to up to two
// outputs. Each 128-byte-wide column chunk goes registers -> 128B-swizzled staging buffer
// -> TMA store of a [32 rows x 128 B] box; two staging buffers alternate.
__device__ __forceinline__ void drain(uint32_t tmem_acc, int q, int lane, uint32_t staging,
                                      uint32_t& chunk_ctr, const Params& p, int m0, int n0,
                                      const CUtensorMap* t0, const CUtensorMap* t1, void* p0,
                                      void* p1) {
  // output chunks of 128 bytes per row: fp32 32 columns, bf16 64 columns, SwiGLU 64
  // output columns from 128 accumulator columns; a tile width that is not a whole number of
  // chunks leaves a tail of tail_cols accumulator columns
  const int chunk_cols = (p.out_f32 || p.epi == EPI_RESIDUAL) ? 32 : 64;
  const int nchunks = p.epi == EPI_SWIGLU ? 2 : p.bn / chunk_cols;
  const int tail_cols = p.epi == EPI_SWIGLU ? 0 : p.bn - nchunks * chunk_cols;
  const uint32_t lane_taddr = tmem_acc + (static_cast<uint32_t>(q * 32) << 16);
  const int y = m0 + q * 32;
  if (p.epi == EPI_ROPE) {
    drain_rope(lane_taddr, lane, staging, p, y, n0, t0, t1);
    return;
  }
  if (p.epi == EPI_LOGSOFTMAX) {
    drain_logsoftmax(lane_taddr, lane, p, y, n0, p0, p1);
    return;
  }
  for (int c = 0; c < nchunks; ++c) {
    const uint32_t buf = staging + (chunk_ctr & 1u) * STAGING_BYTES;
    if (lane == 0) bulk_wait_read1();  // the store issued two chunks ago has read `buf`
    __syncwarp();
    uint32_t w[32];
    int x;
    if (p.epi == EPI_SWIGLU) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        uint32_t g[32], u[32];
        tc_ld_32x32b_x32(lane_taddr + c * 64 + h * 32, g);
        tc_ld_32x32b_x32(lane_taddr + BN / 2 + c * 64 + h * 32, u);
        tc_wait_ld();
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const float g0 = bf16_round(__uint_as_float(g[2 * i]));
          const float g1 = bf16_round(__uint_as_float(g[2 * i + 1]));
          const float u0 = bf16_round(__uint_as_float(u[2 * i]));
          const float u1 = bf16_round(__uint_as_float(u[2 * i + 1]));
          w[h * 16 + i] = pack_bf16x2(g0 / (1.0f + expf(-g0)) * u0, g1 / (1.0f + expf(-g1)) * u1);
        }
      }
      x = n0 / 2 + c * 64;
    } else if (p.epi == EPI_RESIDUAL) {
      tc_ld_32x32b_x32(lane_taddr + c * 32, w);
      tc_wait_ld();
#pragma unroll
      for (int i = 0; i < 32; ++i) w[i] = __float_as_uint(bf16_round(__uint_as_float(w[i])));
      x = n0 + c * 32;
    } else if (p.out_f32) {
      tc_ld_32x32b_x32(lane_taddr + c * 32, w);
      tc_wait_ld();
      x = n0 + c * 32;
    } else {
      uint32_t v0[32], v1[32];
      tc_ld_32x32b_x32(lane_taddr + c * 64, v0);
      tc_ld_32x32b_x32(lane_taddr + c * 64 + 32, v1);
      tc_wait_ld();
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        w[i] = pack_bf16x2(__uint_as_float(v0[2 * i]), __uint_as_float(v0[2 * i + 1]));
        w[16 + i] = pack_bf16x2(__uint_as_float(v1[2 * i]), __uint_as_float(v1[2 * i + 1]));
      }
      x = n0 + c * 64;
    }
    const uint32_t row = buf + lane * 128;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      st_shared_v4(row + ((j ^ (lane & 7)) << 4), w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
    }
    fence_async_smem();
    __syncwarp();
    if (lane == 0) {
      const int n_out = p.epi == EPI_SWIGLU ? p.N / 2 : p.N;
      if (x < n_out && y < p.M) {
        if (p.epi == EPI_RESIDUAL) {
          if (t0) tma_reduce_add_2d(t0, buf, x, y);
          if (t1) tma_reduce_add_2d(t1, buf, x, y);
        } else {
          if (t0) tma_store_2d(t0, buf, x, y);
          if (t1) tma_store_2d(t1, buf, x, y);
        }
      }
      bulk_commit();
    }
    ++chunk_ctr;
  }
  // the tail (a multiple of 16 columns) goes straight from registers to global memory: thread
  // `lane` owns output row y + lane; only this tile writes these columns
  const int row = y + lane;
  for (int c16 = 0; c16 < tail_cols; c16 += 16) {
    uint32_t v[16];
    tc_ld_32x32b_x16(lane_taddr + nchunks * chunk_cols + c16, v);
    tc_wait_ld();
    const int xc = n0 + nchunks * chunk_cols + c16;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int x = xc + 8 * h;
      if (row >= p.M || x >= p.N) continue;  // N % 8 == 0: 8 columns are all in or all out
      const size_t off = static_cast<size_t>(row) * p.N + x;
#pragma unroll
      for (int o = 0; o < 2; ++o) {
        void* dst = o == 0 ? p0 : p1;
        if (dst == nullptr) continue;
        if (p.epi == EPI_RESIDUAL || p.out_f32) {
          float4* d4 = reinterpret_cast<float4*>(static_cast<float*>(dst) + off);
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            float4 val = make_float4(__uint_as_float(v[8 * h + 4 * e]), __uint_as_float(v[8 * h + 4 * e + 1]),
                                     __uint_as_float(v[8 * h + 4 * e + 2]), __uint_as_float(v[8 * h + 4 * e + 3]));
            if (p.epi == EPI_RESIDUAL) {
              const float4 old = d4[e];
              val = make_float4(old.x + bf16_round(val.x), old.y + bf16_round(val.y),
                                old.z + bf16_round(val.z), old.w + bf16_round(val.w));
            }
            d4[e] = val;
          }
        } else {
          uint4 w4;
          w4.x = pack_bf16x2(__uint_as_float(v[8 * h]), __uint_as_float(v[8 * h + 1]));
          w4.y = pack_bf16x2(__uint_as_float(v[8 * h + 2]), __uint_as_float(v[8 * h + 3]));
          w4.z = pack_bf16x2(__uint_as_float(v[8 * h + 4]), __uint_as_float(v[8 * h + 5]));
          w4.w = pack_bf16x2(__uint_as_float(v[8 * h + 6]), __uint_as_float(v[8 * h + 7]));
          *reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(dst) + off) = w4;
        }
      }
    }
  }
}

__global__ void __launch_bounds__(NUM_THREADS, 1)
    dual_lora_gemm_kernel(const __grid_constant__ Maps mp, const Params p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* staging_base = smem + STAGES * STAGE_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(staging_base + EPI_WARPS * 2 * STAGING_BYTES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + NUM_BARS);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int n_local = (p.total_tiles - static_cast<int>(blockIdx.x) + static_cast<int>(gridDim.x) - 1) /
                      static_cast<int>(gridDim.x);
  const int defer_at = min(DEFER, p.kb_main) - 1;

  const uint32_t smem_base = smem_u32(smem);
  auto full_bar = [&](int s) { return smem_u32(&bars[s]); };
  auto empty_bar = [&](int s) { return smem_u32(&bars[STAGES + s]); };
  auto acc_full = [&](int b) { return smem_u32(&bars[2 * STAGES + b]); };
  auto acc_mid = [&](int b) { return smem_u32(&bars[2 * STAGES + 2 + b]); };
  auto acc_empty = [&](int b) { return smem_u32(&bars[2 * STAGES + 4 + b]); };
  const uint32_t mma_done = smem_u32(&bars[2 * STAGES + 6]);

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(acc_full(b), 1);
      mbar_init(acc_mid(b), 32 * EPI_WARPS);
      mbar_init(acc_empty(b), 32 * EPI_WARPS);
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer (whole warp)
    if (elect_one()) {
      for (int i = 0; i < 3; ++i) tma_prefetch_desc(&mp.x[i]);
      tma_prefetch_desc(&mp.w);
      for (int i = 0; i < 2; ++i) {
        tma_prefetch_desc(&mp.u[i]);
        tma_prefetch_desc(&mp.b[i]);
      }
    }
    __syncwarp();
    int it = 0;
    bool ok = true;
    auto load = [&](const CUtensorMap* ma, int xa, int ya, const CUtensorMap* mb, int xb, int yb) {
      const int s = it % STAGES;
      const uint32_t ph = (it / STAGES) & 1;
      if (!warp_wait_bounded(empty_bar(s), ph ^ 1, abort_flag, p.err, kDevTimeoutProducer)) {
        ok = false;
        return;
      }
      if (elect_one()) {
        mbar_arrive_expect_tx(full_bar(s), STAGE_BYTES);
        const uint32_t a_dst = smem_base + s * STAGE_BYTES;
        tma_load_2d(a_dst, ma, xa, ya, full_bar(s));
        tma_load_2d(a_dst + A_TILE, mb, xb, yb, full_bar(s));
      }
      __syncwarp();
      ++it;
    };
    Tile prev{0, 0, 0, 0};
    for (int j = 0; j < n_local && ok; ++j) {
      const Tile tl = decode(p, blockIdx.x + j * gridDim.x);
      const CUtensorMap* tmx = &mp.x[tl.stream];
      for (int kb = 0; kb < p.kb_main && ok; ++kb) {
        load(tmx, kb * BK, tl.m0, &mp.w, kb * BK, tl.n0);
        if (p.deferred && j > 0 && kb == defer_at)
          for (int kl = 0; kl < prev.n_lora && ok; ++kl)
            load(&mp.u[prev.stream == 2 ? 1 : 0], kl * BK, prev.m0, &mp.b[prev.stream == 2 ? 1 : 0], kl * BK, prev.n0);
      }
      if (!p.deferred)
        for (int kl = 0; kl < tl.n_lora && ok; ++kl)
          load(&mp.u[tl.stream == 2 ? 1 : 0], kl * BK, tl.m0, &mp.b[tl.stream == 2 ? 1 : 0], kl * BK, tl.n0);
      prev = tl;
    }
    if (p.deferred && n_local > 0)
      for (int kl = 0; kl < prev.n_lora && ok; ++kl)
        load(&mp.u[prev.stream == 2 ? 1 : 0], kl * BK, prev.m0, &mp.b[prev.stream == 2 ? 1 : 0], kl * BK, prev.n0);
    // copies still in flight must land before the CTA's shared memory is released
    for (int k = (it > STAGES ? it - STAGES : 0); k < it; ++k) {
      volatile int no_abort = 0;
      warp_wait_bounded(full_bar(k % STAGES), (k / STAGES) & 1, &no_abort, p.err, kDevTimeoutDrain);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (whole warp,
    // one elected lane issues; the same lane issues every MMA and commit, so each commit
    // covers all MMAs before it)
    int it = 0;
    bool ok = true;
    // one ring item: nsub MMAs of K = 16 into the accumulator at `acc`; `then` (if non-zero)
    // is an extra barrier to arrive on once these MMAs are done
    auto consume = [&](uint32_t acc, int nsub, bool first, uint32_t then) {
      const int s = it % STAGES;
      const uint32_t ph = (it / STAGES) & 1;
      if (!warp_wait_bounded(full_bar(s), ph, abort_flag, p.err, kDevTimeoutMma)) {
        ok = false;
        return;
      }
      tc_fence_after();
      if (elect_one()) {
        const uint32_t a_base = smem_base + s * STAGE_BYTES;
        const uint32_t b_base = a_base + A_TILE;
        for (int k = 0; k < nsub; ++k)
          tc_mma_bf16(acc, smem_desc_sw128(a_base + k * 32), smem_desc_sw128(b_base + k * 32),
                      IDESC, (first && k == 0) ? 0u : 1u);
        tc_commit(empty_bar(s));
        if (then) tc_commit(then);
      }
      __syncwarp();
      ++it;
    };
    auto lora_nsub = [&](int kl) { return min(BK / 16, (p.r - kl * BK + 15) / 16); };
    auto lora_items = [&](int jj, int n_lora, bool wait_mid) {
      const int b = jj & 1;
      if (wait_mid) {
        if (!warp_wait_bounded(acc_mid(b), (jj >> 1) & 1, abort_flag, p.err, kDevTimeoutMma)) {
          ok = false;
          return;
        }
        tc_fence_after();
      }
      for (int kl = 0; kl < n_lora && ok; ++kl)
        consume(tmem_base + b * 256, lora_nsub(kl), false, kl == n_lora - 1 ? acc_full(b) : 0u);
    };
    Tile prev{0, 0, 0, 0};
    for (int j = 0; j < n_local && ok; ++j) {
      const Tile tl = decode(p, blockIdx.x + j * gridDim.x);
      const int b = j & 1;
      if (!warp_wait_bounded(acc_empty(b), ((j >> 1) & 1) ^ 1, abort_flag, p.err, kDevTimeoutMma))
        break;
      tc_fence_after();
      const uint32_t acc = tmem_base + b * 256;
      for (int kb = 0; kb < p.kb_main && ok; ++kb) {
        const bool last = kb == p.kb_main - 1 && (p.deferred || tl.n_lora == 0);
        consume(acc, BK / 16, kb == 0, last ? acc_full(b) : 0u);
        if (p.deferred && j > 0 && kb == defer_at && ok) lora_items(j - 1, prev.n_lora, true);
      }
      if (!p.deferred && tl.n_lora > 0 && ok) lora_items(j, tl.n_lora, false);
      prev = tl;
    }
    if (p.deferred && n_local > 0 && ok) lora_items(n_local - 1, prev.n_lora, true);
    // every issued MMA has finished before TMEM is released
    if (elect_one()) tc_commit(mma_done);
    __syncwarp();
    volatile int no_abort = 0;
    warp_wait_bounded(mma_done, 0, &no_abort, p.err, kDevTimeoutDrain);
  } else {
    // -------------------------------------------------------------- epilogue
    const int q = warp & 3;
    const uint32_t staging = smem_u32(staging_base) + (warp - 2) * 2 * STAGING_BYTES;
    uint32_t chunk_ctr = 0;
    const CUtensorMap* y_off = p.has_off ? &mp.y[0] : nullptr;
    const CUtensorMap* y_on = p.has_on ? &mp.y[1] : nullptr;
    const CUtensorMap* y_crit = p.has_crit ? &mp.y[2] : nullptr;
    void* py_off = p.has_off ? p.y_off_ptr : nullptr;
    void* py_on = p.has_on ? p.y_on_ptr : nullptr;
    void* py_crit = p.has_crit ? p.y_crit_ptr : nullptr;
    if (lane == 0) {
      for (int i = 0; i < 3; ++i) tma_prefetch_desc(&mp.y[i]);
    }
    for (int j = 0; j < n_local; ++j) {
      const Tile tl = decode(p, blockIdx.x + j * gridDim.x);
      const int b = j & 1;
      const uint32_t acc = tmem_base + b * 256;
      if (p.deferred) {
        if (!mbar_wait_bounded(acc_full(b), 0, abort_flag, p.err, kDevTimeoutEpilogue)) break;
        tc_fence_after();
        drain(acc, q, lane, staging, chunk_ctr, p, tl.m0, tl.n0, y_off, nullptr, py_off, nullptr);
        tc_fence_before();
        mbar_arrive(acc_mid(b));
        if (!mbar_wait_bounded(acc_full(b), 1, abort_flag, p.err, kDevTimeoutEpilogue)) break;
        tc_fence_after();
        drain(acc, q, lane, staging, chunk_ctr, p, tl.m0, tl.n0, y_on, nullptr, py_on, nullptr);
      } else {
        if (!mbar_wait_bounded(acc_full(b), (j >> 1) & 1, abort_flag, p.err, kDevTimeoutEpilogue))
          break;
        tc_fence_after();
        if (p.shared_x)
          drain(acc, q, lane, staging, chunk_ctr, p, tl.m0, tl.n0, tl.n_lora > 0 ? nullptr : y_off, y_on,
                tl.n_lora > 0 ? nullptr : py_off, py_on);
        else
          drain(acc, q, lane, staging, chunk_ctr, p, tl.m0, tl.n0,
                tl.stream == 0 ? y_off : (tl.stream == 1 ? y_on : y_crit), nullptr,
                tl.stream == 0 ? py_off : (tl.stream == 1 ? py_on : py_crit), nullptr);
      }
      tc_fence_before();
      mbar_arrive(acc_empty(b));
    }
    if (lane == 0) bulk_wait_all();
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}


// ============================================================================================
// Two-CTA variant (tcgen05 cta_group::2): a cluster of two CTAs on two SMs computes a
// 256 x 256 tile with one M = 256 MMA stream issued by the leader CTA (cluster rank 0).
// Each CTA holds its 128 rows of A and 128 of the 256 rows of B, so a pair moves half the
// B bytes of two independent 128 x 256 tiles, and a 32 KiB stage allows a 6-deep ring per
// SM. Each CTA's TMEM holds the accumulator rows of its own 128 output rows; each CTA's
// epilogue drains them. Protocol: both CTAs' TMA loads complete on the leader's full
// barrier (the leader posts the byte count of both); the leader's MMA commits arrive on
// the empty / accumulator barriers of both CTAs (multicast); both CTAs' epilogue warps
// arrive on the leader's accumulator-drained barriers.
constexpr int STAGES2 = 6;
constexpr int B_HALF = 128 * BK * 2;             // 16 KiB: this CTA's 128 rows of B
constexpr int STAGE2_BYTES = A_TILE + B_HALF;     // 32 KiB
constexpr int SMEM2_BYTES =
    1024 + STAGES2 * STAGE2_BYTES + EPI_WARPS * 2 * STAGING_BYTES + (2 * STAGES2 + 7) * 8 + 16;

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(NUM_THREADS, 1)
    dual_lora_gemm_2cta_kernel(const __grid_constant__ Maps mp, const Params p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* staging_base = smem + STAGES2 * STAGE2_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(staging_base + EPI_WARPS * 2 * STAGING_BYTES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES2 + 7);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const bool leader = rank == 0;
  const int cluster = static_cast<int>(blockIdx.x >> 1);
  const int nclusters = static_cast<int>(gridDim.x >> 1);
  const int n_local = (p.total_tiles - cluster + nclusters - 1) / nclusters;
  const int defer_at = min(DEFER, p.kb_main) - 1;

  const uint32_t smem_base = smem_u32(smem);
  auto full_bar = [&](int s) { return smem_u32(&bars[s]); };
  auto empty_bar = [&](int s) { return smem_u32(&bars[STAGES2 + s]); };
  auto acc_full = [&](int b) { return smem_u32(&bars[2 * STAGES2 + b]); };
  auto acc_mid = [&](int b) { return smem_u32(&bars[2 * STAGES2 + 2 + b]); };
  auto acc_empty = [&](int b) { return smem_u32(&bars[2 * STAGES2 + 4 + b]); };
  const uint32_t mma_done = smem_u32(&bars[2 * STAGES2 + 6]);

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES2; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(acc_full(b), 1);
      mbar_init(acc_mid(b), 2 * EPI_WARPS);
      mbar_init(acc_empty(b), 2 * EPI_WARPS);
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // barriers of both CTAs are initialised before any remote signal
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  // tile -> (stream, 256-row block, column block); this CTA's rows are m0 + 128 rank
  auto decode2 = [&](int t) {
    Tile tl;
    tl.stream = t % p.streams;
    t /= p.streams;
    int mi, ni;
    if (p.m_group > 0) {
      const int per_group = p.m_group * p.n_tiles;
      const int grp = t / per_group, r = t - grp * per_group;
      const int gm = min(p.m_group, p.m_tiles - grp * p.m_group);  // the last group may be short
      mi = grp * p.m_group + r % gm;
      ni = r / gm;
    } else {
      mi = t % p.m_tiles;
      ni = t / p.m_tiles;
    }
    tl.m0 = mi * 256 + static_cast<int>(rank) * 128;
    tl.n0 = ni * p.bn;
    const bool lora = p.shared_x ? true : (tl.stream >= 1);
    const bool wanted = tl.stream == 2 ? p.has_crit : p.has_on;
    tl.n_lora = (p.kb_lora > 0 && lora && wanted) ? p.kb_lora : 0;
    return tl;
  };

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer (both CTAs;
    // whole warp, one elected lane issues)
    int it = 0;
    bool ok = true;
    const uint32_t leader_full0 = map_to_rank(full_bar(0), 0);
    auto load = [&](const CUtensorMap* ma, int xa, int ya, const CUtensorMap* mb, int xb, int yb) {
      const int s = it % STAGES2;
      const uint32_t ph = (it / STAGES2) & 1;
      if (!warp_wait_bounded(empty_bar(s), ph ^ 1, abort_flag, p.err, kDevTimeoutProducer)) {
        ok = false;
        return;
      }
      if (elect_one()) {
        if (leader) mbar_arrive_expect_tx(full_bar(s), 2 * (A_TILE + p.bn * 64));
        const uint32_t bar = leader_full0 + s * 8;
        const uint32_t a_dst = smem_base + s * STAGE2_BYTES;
        tma_load_2d_pair(a_dst, ma, xa, ya, bar);
        tma_load_2d_pair(a_dst + A_TILE, mb, xb, yb, bar);
      }
      __syncwarp();
      ++it;
    };
    const int brow = static_cast<int>(rank) * (p.bn / 2);  // this CTA's half of the B rows
    Tile prev{0, 0, 0, 0};
    for (int j = 0; j < n_local && ok; ++j) {
      const Tile tl = decode2(cluster + j * nclusters);
      const CUtensorMap* tmx = &mp.x[tl.stream];
      for (int kb = 0; kb < p.kb_main && ok; ++kb) {
        load(tmx, kb * BK, tl.m0, &mp.w, kb * BK, tl.n0 + brow);
        if (p.deferred && j > 0 && kb == defer_at)
          for (int kl = 0; kl < prev.n_lora && ok; ++kl)
            load(&mp.u[prev.stream == 2 ? 1 : 0], kl * BK, prev.m0, &mp.b[prev.stream == 2 ? 1 : 0], kl * BK, prev.n0 + brow);
      }
      if (!p.deferred)
        for (int kl = 0; kl < tl.n_lora && ok; ++kl)
          load(&mp.u[tl.stream == 2 ? 1 : 0], kl * BK, tl.m0, &mp.b[tl.stream == 2 ? 1 : 0], kl * BK, tl.n0 + brow);
      prev = tl;
    }
    if (p.deferred && n_local > 0)
      for (int kl = 0; kl < prev.n_lora && ok; ++kl)
        load(&mp.u[prev.stream == 2 ? 1 : 0], kl * BK, prev.m0, &mp.b[prev.stream == 2 ? 1 : 0], kl * BK, prev.n0 + brow);
    // this CTA's copies in flight must land before its shared memory is released: the
    // stage's empty barrier (committed after the MMAs that read it) covers them
    for (int k = (it > STAGES2 ? it - STAGES2 : 0); k < it; ++k) {
      volatile int no_abort = 0;
      warp_wait_bounded(empty_bar(k % STAGES2), (k / STAGES2) & 1, &no_abort, p.err,
                        kDevTimeoutDrain);
    }
  } else if (warp == 1) {
    if (leader) {
      // ---------------------------------------------------------- MMA issuer (leader CTA;
      // whole warp, one elected lane issues every MMA and commit)
      const uint32_t idesc2 = idesc_bf16_f32(256, p.bn);
      int it = 0;
      bool ok = true;
      auto consume = [&](uint32_t acc, int nsub, bool first, uint32_t then) {
        const int s = it % STAGES2;
        const uint32_t ph = (it / STAGES2) & 1;
        if (!warp_wait_bounded(full_bar(s), ph, abort_flag, p.err, kDevTimeoutMma)) {
          ok = false;
          return;
        }
        tc_fence_after();
        if (elect_one()) {
          const uint32_t a_base = smem_base + s * STAGE2_BYTES;
          const uint32_t b_base = a_base + A_TILE;
          for (int k = 0; k < nsub; ++k)
            tc_mma2_bf16(acc, smem_desc_sw128(a_base + k * 32), smem_desc_sw128(b_base + k * 32),
                         idesc2, (first && k == 0) ? 0u : 1u);
          tc_commit_pair(empty_bar(s));
          if (then) tc_commit_pair(then);
        }
        __syncwarp();
        ++it;
      };
      auto lora_nsub = [&](int kl) { return min(BK / 16, (p.r - kl * BK + 15) / 16); };
      auto lora_items = [&](int jj, int n_lora, bool wait_mid) {
        const int b = jj & 1;
        if (wait_mid) {
          if (!warp_wait_cluster_bounded(acc_mid(b), (jj >> 1) & 1, abort_flag, p.err,
                                         kDevTimeoutMma)) {
            ok = false;
            return;
          }
          tc_fence_after();
        }
        for (int kl = 0; kl < n_lora && ok; ++kl)
          consume(tmem_base + b * 256, lora_nsub(kl), false, kl == n_lora - 1 ? acc_full(b) : 0u);
      };
      Tile prev{0, 0, 0, 0};
      for (int j = 0; j < n_local && ok; ++j) {
        const Tile tl = decode2(cluster + j * nclusters);
        const int b = j & 1;
        if (!warp_wait_cluster_bounded(acc_empty(b), ((j >> 1) & 1) ^ 1, abort_flag, p.err,
                                       kDevTimeoutMma))
          break;
        tc_fence_after();
        const uint32_t acc = tmem_base + b * 256;
        for (int kb = 0; kb < p.kb_main && ok; ++kb) {
          const bool last = kb == p.kb_main - 1 && (p.deferred || tl.n_lora == 0);
          consume(acc, BK / 16, kb == 0, last ? acc_full(b) : 0u);
          if (p.deferred && j > 0 && kb == defer_at && ok) lora_items(j - 1, prev.n_lora, true);
        }
        if (!p.deferred && tl.n_lora > 0 && ok) lora_items(j, tl.n_lora, false);
        prev = tl;
      }
      if (p.deferred && n_local > 0 && ok) lora_items(n_local - 1, prev.n_lora, true);
      if (elect_one()) tc_commit_pair(mma_done);
      __syncwarp();
      volatile int no_abort = 0;
      warp_wait_bounded(mma_done, 0, &no_abort, p.err, kDevTimeoutDrain);
    }
  } else {
    // -------------------------------------------------------------- epilogue (both CTAs)
    const int q = warp & 3;
    const uint32_t staging = smem_u32(staging_base) + (warp - 2) * 2 * STAGING_BYTES;
    uint32_t chunk_ctr = 0;
    const CUtensorMap* y_off = p.has_off ? &mp.y[0] : nullptr;
    const CUtensorMap* y_on = p.has_on ? &mp.y[1] : nullptr;
    const CUtensorMap* y_crit = p.has_crit ? &mp.y[2] : nullptr;
    void* py_off = p.has_off ? p.y_off_ptr : nullptr;
    void* py_on = p.has_on ? p.y_on_ptr : nullptr;
    void* py_crit = p.has_crit ? p.y_crit_ptr : nullptr;
    const uint32_t leader_mid0 = map_to_rank(acc_mid(0), 0);
    const uint32_t leader_empty0 = map_to_rank(acc_empty(0), 0);
    auto signal = [&](uint32_t leader_bar0, int b) {
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(leader_bar0 + b * 8);
    };
    for (int j = 0; j < n_local; ++j) {
      const Tile tl = decode2(cluster + j * nclusters);
      const int b = j & 1;
      const uint32_t acc = tmem_base + b * 256;
      if (p.deferred) {
        if (!mbar_wait_bounded(acc_full(b), 0, abort_flag, p.err, kDevTimeoutEpilogue)) break;
        tc_fence_after();
        drain(acc, q, lane, staging, chunk_ctr, p, tl.m0, tl.n0, y_off, nullptr, py_off, nullptr);
        tc_fence_before();
        signal(leader_mid0, b);
        if (!mbar_wait_bounded(acc_full(b), 1, abort_flag, p.err, kDevTimeoutEpilogue)) break;
        tc_fence_after();
        drain(acc, q, lane, staging, chunk_ctr, p, tl.m0, tl.n0, y_on, nullptr, py_on, nullptr);
      } else {
        if (!mbar_wait_bounded(acc_full(b), (j >> 1) & 1, abort_flag, p.err, kDevTimeoutEpilogue))
          break;
        tc_fence_after();
        if (p.shared_x)
          drain(acc, q, lane, staging, chunk_ctr, p, tl.m0, tl.n0, tl.n_lora > 0 ? nullptr : y_off, y_on,
                tl.n_lora > 0 ? nullptr : py_off, py_on);
        else
          drain(acc, q, lane, staging, chunk_ctr, p, tl.m0, tl.n0,
                tl.stream == 0 ? y_off : (tl.stream == 1 ? y_on : y_crit), nullptr,
                tl.stream == 0 ? py_off : (tl.stream == 1 ? py_on : py_crit), nullptr);
      }
      tc_fence_before();
      signal(leader_empty0, b);
    }
    if (lane == 0) bulk_wait_all();
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // no CTA leaves while its peer may still touch its barriers or smem
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(TMEM_COLS)
                 : "memory");
  }
}

}  // namespace tcgemm

// ------------------------------------------------------------------ host side

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (fn == nullptr) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  }
  return fn;
}

// 2-D tensor map over a row-major [rows, cols] matrix with row stride ld elements, 128-byte
// swizzle and a box of [box_rows, 128 bytes]; out-of-bounds loads read zero, out-of-bounds
// stores are dropped.
bool make_tma_map(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int64_t ld,
                  int box_rows, bool f32) {
  EncodeTiledFn enc = get_encode_fn();
  if (enc == nullptr) return false;
  const int esize = f32 ? 4 : 2;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * esize};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(128 / esize), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                   const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                   CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool make_tma_map_3d(CUtensorMap* map, const void* base, int64_t cols, int64_t rows,
                     int64_t planes, int64_t ld, int64_t plane_stride, int box_rows) {
  EncodeTiledFn enc = get_encode_fn();
  if (enc == nullptr) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows),
                        static_cast<cuuint64_t>(planes)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(ld) * 2, static_cast<cuuint64_t>(plane_stride) * 2};
  cuuint32_t box[3] = {64, static_cast<cuuint32_t>(box_rows), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
                   box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

static bool make_map(CUtensorMap* map, const void* base, int64_t rows, int64_t cols,
                     int box_rows, bool f32) {
  return make_tma_map(map, base, rows, cols, cols, box_rows, f32);
}

static int sm_count() {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  if (cached[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    cached[dev] = n;
  }
  return cached[dev];
}

// Tile width of the CTA-pair kernel: the candidate with the least waves x (width + 224)
// over the clusters. A tile costs its columns plus a fixed share worth about 224 columns
// (fitted on GB300: 6144 x 4096 x 12288 ran 6.8 % slower at 208 wide, 19 full waves, than at
// 256, 15.2 waves). Narrower tiles pay off when they turn a nearly empty last wave into
// full ones (4096 output columns at 3072 rows per stream: 256 wide gives 5.05 waves, 224
// wide exactly 6; measured +8 %). The SwiGLU epilogue needs 256 (128 gate + 128 up).
static int pick_tile_width(const GemmArgs& a, int nclusters) {
  if (a.epi == tcgemm::EPI_SWIGLU || a.epi == tcgemm::EPI_ROPE || a.epi == tcgemm::EPI_LOGSOFTMAX ||
      nclusters < 1)
    return 256;
  const int64_t m_tiles = (a.M + 255) / 256;
  const int64_t streams = a.shared_x ? 1 : (a.x_crit != nullptr ? 3 : 2);
  int best = 256;
  int64_t best_cost = INT64_MAX;
  for (int bn : {256, 240, 224, 208, 192}) {
    const int64_t tiles = m_tiles * streams * ((a.N + bn - 1) / bn);
    const int64_t waves = (tiles + nclusters - 1) / nclusters;
    const int64_t cost = waves * (bn + 224);
    if (cost < best_cost) {
      best = bn;
      best_cost = cost;
    }
  }
  return best;
}

int launch_dual_lora_gemm_tc(const GemmArgs& a, cudaStream_t stream) {
  using namespace tcgemm;
  static bool attr_set = false;
  if (!attr_set) {
    if (cudaFuncSetAttribute(dual_lora_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             SMEM_BYTES) != cudaSuccess)
      return -1;
    if (cudaFuncSetAttribute(dual_lora_gemm_2cta_kernel,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM2_BYTES) != cudaSuccess)
      return -1;
    attr_set = true;
  }
  const int nsm = sm_count();
  if (nsm <= 0) return -1;
  // 256-row CTA pairs once every stream has more than one 128-row tile of work
  const bool pair = a.M > BM && nsm >= 2 && !a.single_cta;
  const int bn = pair ? pick_tile_width(a, nsm / 2) : BN;
  const bool tri = a.x_crit != nullptr && !a.shared_x;  // off, on and critic streams
  Maps mp;
  const bool lora = a.r > 0;
  const bool f32 = a.out_f32 != 0;
  if (!make_map(&mp.x[0], a.x_off, a.M, a.K, BM, false)) return -2;
  if (!make_map(&mp.x[1], a.shared_x ? a.x_off : a.x_on, a.M, a.K, BM, false)) return -2;
  if (!make_map(&mp.x[2], tri ? a.x_crit : a.x_off, a.M, a.K, BM, false)) return -2;
  const int brows = pair ? bn / 2 : BN;  // a CTA of a pair loads half of the tile's W rows
  if (!make_map(&mp.w, a.W, a.N, a.K, brows, false)) return -2;
  for (int i = 0; i < 2; ++i) {
    const void* u = i == 0 ? a.u : a.u_crit;
    const void* B = i == 0 ? a.B : a.B_crit;
    if (lora && u != nullptr && B != nullptr) {
      if (!make_map(&mp.u[i], u, a.M, a.r, BM, false)) return -2;
      if (!make_map(&mp.b[i], B, a.N, a.r, brows, false)) return -2;
    } else {  // never read
      mp.u[i] = mp.x[0];
      mp.b[i] = mp.w;
    }
  }
  const void* any_y = a.y_off ? a.y_off : (a.y_on ? a.y_on : a.y_crit);
  // output tensor: SwiGLU writes bf16 [M, N/2]; the residual mode adds into fp32 [M, N]
  const int64_t n_out = a.epi == tcgemm::EPI_SWIGLU ? a.N / 2 : a.N;
  const bool out32 = a.epi == tcgemm::EPI_RESIDUAL ? true : (a.epi == tcgemm::EPI_SWIGLU ? false : f32);
  for (int i = 0; i < 3; ++i) {
    void* y = i == 0 ? a.y_off : (i == 1 ? a.y_on : a.y_crit);
    if (a.epi == tcgemm::EPI_LOGSOFTMAX) {  // no per-column outputs: the maps are never used
      mp.y[i] = mp.x[0];
    } else if (!make_map(&mp.y[i], y ? y : any_y, a.M, n_out, 32, out32)) {
      return -2;
    }
  }

  Params p;
  p.M = static_cast<int>(a.M);
  p.N = static_cast<int>(a.N);
  p.K = static_cast<int>(a.K);
  p.epi = a.epi;
  p.kb_main = static_cast<int>((a.K + BK - 1) / BK);
  p.kb_lora = lora ? static_cast<int>((a.r + BK - 1) / BK) : 0;
  p.r = static_cast<int>(a.r);
  p.shared_x = a.shared_x ? 1 : 0;
  p.has_off = a.y_off != nullptr;
  p.has_on = a.y_on != nullptr;
  p.has_crit = tri && a.y_crit != nullptr && (!lora || (a.u_crit != nullptr && a.B_crit != nullptr));
  p.deferred = (p.shared_x && lora && p.has_off && p.has_on) ? 1 : 0;
  p.streams = a.shared_x ? 1 : (tri ? 3 : 2);
  p.m_tiles = static_cast<int>(pair ? (a.M + 255) / 256 : (a.M + BM - 1) / BM);
  p.n_tiles = static_cast<int>((a.N + bn - 1) / bn);
  p.total_tiles = p.m_tiles * p.n_tiles * p.streams;
  // Tile order of the CTA-pair kernel. Over all of M, the tiles in flight at once (one per
  // pair) cover every m-tile of a few n-columns: x stays in L2 if it fits, else it is read
  // again for each column (a 3072 x 11008 down-projection input of both streams, 135 MB,
  // measured 1026 MB of DRAM reads per launch). Beyond half of L2, m-tiles go in groups
  // whose inputs total about 48 MB, and W is read once per group instead. From 40 MB of
  // input (the 50 MB q/k/v, o and gate/up inputs of both streams), groups of about 24 MB:
  // x then stays while W is read twice (measured DRAM reads per launch: q/k/v 336 -> 280 MB,
  // o 252 -> 235 MB, gate/up 457 -> 436 MB; groups of 12 MB re-read W too often).
  p.m_group = 0;
  if (pair) {
    const int64_t x_bytes = static_cast<int64_t>(p.streams) * a.M * a.K * 2;
    const int64_t mtile_bytes = static_cast<int64_t>(p.streams) * 256 * a.K * 2;
    if (x_bytes > (int64_t{40} << 20) && p.m_tiles > 1) {
      const int64_t budget = x_bytes > (int64_t{64} << 20) ? (int64_t{48} << 20) : (int64_t{24} << 20);
      const int64_t g = budget / mtile_bytes;
      p.m_group = static_cast<int>(g < 1 ? 1 : (g > p.m_tiles ? p.m_tiles : g));
      if (p.m_group >= p.m_tiles) p.m_group = 0;
    }
  }
  p.out_f32 = a.out_f32;
  p.bn = bn;
  p.rope_P = static_cast<int>(a.rope_P < 1 ? 1 : a.rope_P);
  p.rope_cols = static_cast<int>(a.rope_cols);
  p.rope_table = static_cast<const float2*>(a.rope_table);
  p.lsm_target = a.lsm_target;
  p.lsm_ids = a.lsm_ids;
  p.lsm_L = static_cast<int>(a.lsm_L < 1 ? 1 : a.lsm_L);
  p.lsm_ids_ld = static_cast<int>(a.lsm_ids_ld);
  p.lsm_ids_off = static_cast<int>(a.lsm_ids_off);
  p.y_off_ptr = a.y_off;
  p.y_on_ptr = a.y_on;
  p.y_crit_ptr = a.y_crit;
  p.err = a.err;
  if (pair) {
    const int nclusters = nsm / 2;
    const unsigned grid =
        2u * static_cast<unsigned>(p.total_tiles < nclusters ? p.total_tiles : nclusters);
    dual_lora_gemm_2cta_kernel<<<grid, NUM_THREADS, SMEM2_BYTES, stream>>>(mp, p);
    return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
  }
  const unsigned grid = static_cast<unsigned>(p.total_tiles < nsm ? p.total_tiles : nsm);
  dual_lora_gemm_kernel<<<grid, NUM_THREADS, SMEM_BYTES, stream>>>(mp, p);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace hydra
