// Skinny LoRA kernels:
//  * lora_down: u = s * (x_on A^T), bf16 [M, r]; the rank-r down-projection of the
//    LoRA update (§2 Stage 3: LoRA on all linear layers), with the scale folded in fp32
//    before the bf16 rounding. It is the operand of the LoRA-up MMA of the tcgen05
//    kernel and of the GEMV below. (Uses mma.sync: a skinny product far too narrow for a
//    128-row tcgen05 tile to stay busy.)
//  * dual_lora_gemv: the dual-output linear for decode-shaped inputs (at most 16 token
//    rows over both streams), y_off = x_off W^T, y_on = x_on W^T + u B^T, streaming W once
//    (see the kernel). Used where a 128-row tcgen05 tile would be almost empty.
#include <algorithm>
#include <utility>

#include "common.cuh"
#include "kernels.h"

namespace hydra {
namespace {

// ---------------------------------------------------------------- lora_down
//
// u[M, r] = bf16(s * x A^T) as a skinny matrix product on the tensor cores (mma.sync
// m16n8k16, bf16 in, fp32 accumulate). A thread-block cluster of ck CTAs takes 16 token rows
// and up to 64 ranks and splits K: each CTA's 8 warps split its slice again and reduce their
// partial tiles in shared memory, and CTA rank 0 adds the ck tiles through distributed
// shared memory in rank order (deterministic, no global scratch). The split puts enough
// loads in flight: with one CTA per 16 rows, 2048 rows gave 128 CTAs, 12 % of the warp slots,
// and the kernel waited on memory latency at 14 % of DRAM bandwidth. The contraction over k
// is order-free, so inside each 32-wide chunk of k both operands use the same permutation of
// k: the fragment slots a lane feeds in the chunk's two k-steps are its 8 consecutive
// elements [8c, 8c + 8), which arrive with one 16-byte load per row.

constexpr int kDownWarps = 8;

__device__ __forceinline__ uint4 ld16(const __nv_bfloat16* p, bool ok) {
  return ok ? __ldg(reinterpret_cast<const uint4*>(p)) : make_uint4(0u, 0u, 0u, 0u);
}

__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                               uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

template <int NT>  // NT n-tiles of 8 ranks
__global__ void __launch_bounds__(32 * kDownWarps)
    lora_down_kernel(const __nv_bfloat16* __restrict__ x, int M, int K,
                     const __nv_bfloat16* __restrict__ A, int r, float s,
                     __nv_bfloat16* __restrict__ u, int ck) {
  __shared__ float red[kDownWarps][16][NT * 8 + 1];
  __shared__ float tile[16][NT * 8];  // this CTA's sum over its warps
  pdl_launch_dependents();
  pdl_wait();  // x is written by the preceding kernel
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int g = lane >> 2, c = lane & 3;
  const uint32_t rank = ck > 1 ? cluster_rank() : 0u;
  const int row0 = (blockIdx.x / ck) * 16;
  const int n_base = blockIdx.y * NT * 8;
  // this CTA's K slice, then this warp's part of it, in chunks of 32
  const int nchunk = (K + 31) / 32;
  const int per_cta = (nchunk + ck - 1) / ck;
  const int cta0 = static_cast<int>(rank) * per_cta;
  const int cta1 = min(nchunk, cta0 + per_cta);
  const int per = (max(cta1 - cta0, 0) + kDownWarps - 1) / kDownWarps;
  const int ch0 = cta0 + warp * per;
  const int ch1 = min(cta1, ch0 + per);

  const bool r_lo = row0 + g < M, r_hi = row0 + g + 8 < M;
  const __nv_bfloat16* x_lo = x + static_cast<size_t>(r_lo ? row0 + g : 0) * K + 8 * c;
  const __nv_bfloat16* x_hi = x + static_cast<size_t>(r_hi ? row0 + g + 8 : 0) * K + 8 * c;
  const __nv_bfloat16* a_row[NT];
  bool a_ok[NT];
#pragma unroll
  for (int t = 0; t < NT; ++t) {
    const int n = n_base + t * 8 + g;
    a_ok[t] = n < r;
    a_row[t] = A + static_cast<size_t>(a_ok[t] ? n : 0) * K + 8 * c;
  }
  float d[NT][4];
#pragma unroll
  for (int t = 0; t < NT; ++t) d[t][0] = d[t][1] = d[t][2] = d[t][3] = 0.f;

#pragma unroll 4
  for (int ch = ch0; ch < ch1; ++ch) {
    const int k = ch * 32;
    const bool kv = k + 8 * c < K;  // K % 8 == 0: a lane's 8 elements are all in or all out
    const uint4 xl = ld16(x_lo + k, r_lo && kv);
    const uint4 xh = ld16(x_hi + k, r_hi && kv);
    uint4 bv[NT];
#pragma unroll
    for (int t = 0; t < NT; ++t) bv[t] = ld16(a_row[t] + k, a_ok[t] && kv);
    const uint32_t a0[4] = {xl.x, xh.x, xl.y, xh.y};  // k-step 0: elements 8c .. 8c + 3
    const uint32_t a1[4] = {xl.z, xh.z, xl.w, xh.w};  // k-step 1: elements 8c + 4 .. 8c + 7
#pragma unroll
    for (int t = 0; t < NT; ++t) {
      mma_bf16_16816(d[t], a0, bv[t].x, bv[t].y);
      mma_bf16_16816(d[t], a1, bv[t].z, bv[t].w);
    }
  }
#pragma unroll
  for (int t = 0; t < NT; ++t) {
    red[warp][g][t * 8 + 2 * c] = d[t][0];
    red[warp][g][t * 8 + 2 * c + 1] = d[t][1];
    red[warp][g + 8][t * 8 + 2 * c] = d[t][2];
    red[warp][g + 8][t * 8 + 2 * c + 1] = d[t][3];
  }
  __syncthreads();
  for (int e = threadIdx.x; e < 16 * NT * 8; e += blockDim.x) {
    const int rr = e / (NT * 8), cc = e % (NT * 8);
    float v = 0.f;
#pragma unroll
    for (int w = 0; w < kDownWarps; ++w) v += red[w][rr][cc];
    tile[rr][cc] = v;
  }
  if (ck > 1) cluster_sync_all();  // every CTA's tile is complete and visible
  else __syncthreads();
  if (rank == 0) {
    for (int e = threadIdx.x; e < 16 * NT * 8; e += blockDim.x) {
      const int rr = e / (NT * 8), cc = e % (NT * 8);
      float v = tile[rr][cc];
      for (int q = 1; q < ck; ++q) v += ld_cluster_f32(&tile[rr][cc], static_cast<uint32_t>(q));
      const int m = row0 + rr, n = n_base + cc;
      if (m < M && n < r) u[static_cast<size_t>(m) * r + n] = __float2bfloat16_rn(s * v);
    }
  }
  if (ck > 1) cluster_sync_all();  // rank 0's remote reads end before any CTA exits
}

// cudaLaunchKernelEx with a (ck, 1, 1) cluster (none when ck == 1) and programmatic
// dependent launch
template <typename... KArgs, typename... Args>
cudaError_t launch_down(void (*kernel)(KArgs...), dim3 grid, int ck, cudaStream_t st,
                        Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(32 * kDownWarps);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = static_cast<unsigned>(ck);
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = ck > 1 ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// ---------------------------------------------------------------- lora_down, streaming form
//
// For 64 token rows and more, x is streamed once from HBM by TMA. A thread-block cluster of
// ck CTAs (1, 2, 4 or 8) takes a block of 64 rows and up to 64 ranks and splits K into ck
// contiguous ranges of 64-wide k-blocks. In each CTA one producer warp moves [64 rows x 64 k]
// tiles of x and [8 NT ranks x 64 k] tiles of A through a 6-stage ring (128-byte swizzle);
// each of four consumer warps takes one 16-wide k-step of every stage over all 64 rows
// (ldmatrix, then mma.sync m16n8k16 with fp32 accumulation), so every byte staged in shared
// memory is read once and the arithmetic never holds the stream back. The warps' partial
// [64 x 8 NT] tiles are summed in shared memory in warp order; CTA q finishes rows
// [q 64 / ck, (q + 1) 64 / ck) of the block: every CTA pushes its sums of those rows into
// q's receive buffer with stores to distributed shared memory, one cluster barrier makes them
// visible, and q adds the ck slices in rank order, so the result does not depend on timing
// (a pull through remote loads cost about 2 us more per launch: each remote load waits a
// full round trip). All CTAs of a launch fit on the GPU at once (2-4 per SM), so every load
// of x is issued at the start and the launch costs about one pass over x at HBM speed plus
// the reduction.
namespace lds {

constexpr int kBM = 64;          // token rows per CTA
constexpr int kConsumers = 4;    // consumer warps; warp kConsumers is the producer
constexpr int kThreads = 32 * (kConsumers + 1);
constexpr int kXTile = kBM * 128;  // [64 rows x 64 bf16], 8 KiB

template <int NT>  // NT n-tiles of 8 ranks (1, 2, 4 or 8)
struct Cfg {
  // ring depth: as deep as still lets three CTAs share an SM (two at 64 ranks)
  static constexpr int kStages = NT <= 2 ? 6 : 5;
  static constexpr int kATile = 8 * NT * 128;
  static constexpr int kStage = kXTile + kATile;  // a multiple of 1024: tiles stay aligned
  static constexpr int kRing = kStages * kStage;
  static constexpr int kLd = 8 * NT + 4;          // fp32 row stride of the partial tiles
  static constexpr int kPart = kBM * kLd * 4;
  static_assert(kConsumers * kPart <= kRing, "partial tiles reuse the ring");
  // receive buffer [ck][64 / ck][8 NT] fp32: the cluster's sums of this CTA's rows; outside
  // the ring, since other CTAs may write it while this one still streams
  static constexpr int kRecvOff = kRing;
  static constexpr int kBarOff = kRecvOff + kBM * 8 * NT * 4;
  static constexpr int kSmem = 1024 + kBarOff + 2 * kStages * 8 + 16;
};

__device__ __forceinline__ void st_cluster_v4(const float* local, uint32_t rank, float4 v) {
  uint32_t raddr;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(raddr) : "r"(smem_u32(local)), "r"(rank));
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(raddr), "f"(v.x), "f"(v.y),
               "f"(v.z), "f"(v.w)
               : "memory");
}

__device__ __forceinline__ void store_u4(__nv_bfloat16* u, int r, int m, int nn, float s, float4 v) {
  uint2 o;
  o.x = pack_bf16x2(s * v.x, s * v.y);
  o.y = pack_bf16x2(s * v.z, s * v.w);
  *reinterpret_cast<uint2*>(u + static_cast<size_t>(m) * r + nn) = o;
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&a)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(a[0]), "=r"(a[1]), "=r"(a[2]), "=r"(a[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x2(uint32_t addr, uint32_t (&a)[2]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0,%1}, [%2];"
               : "=r"(a[0]), "=r"(a[1])
               : "r"(addr));
}
// byte offset of 16-byte chunk `chunk` of row `row` in a 128-byte-swizzled tile
__device__ __forceinline__ uint32_t sw128(int row, int chunk) {
  return static_cast<uint32_t>(row * 128 + ((chunk ^ (row & 7)) << 4));
}

template <int NT>
__global__ void __launch_bounds__(kThreads)
    lora_down_stream_kernel(const __grid_constant__ CUtensorMap tm_x,
                            const __grid_constant__ CUtensorMap tm_a, int M, int K, int r, float s,
                            __nv_bfloat16* __restrict__ u, int ck, int* err) {
  using C = Cfg<NT>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::kBarOff);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 2 * C::kStages);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t sbase = smem_u32(smem);
  auto full = [&](int i) { return smem_u32(&bars[i]); };
  auto empty = [&](int i) { return smem_u32(&bars[C::kStages + i]); };

  const uint32_t rank = ck > 1 ? cluster_rank() : 0u;
  const int row0 = static_cast<int>(blockIdx.x / ck) * kBM;
  const int n_base = static_cast<int>(blockIdx.y) * 64;
  const int nkb = (K + 63) / 64;
  const int kb0 = static_cast<int>((static_cast<int64_t>(nkb) * rank) / ck);
  const int kb1 = static_cast<int>((static_cast<int64_t>(nkb) * (rank + 1)) / ck);
  const int n = kb1 - kb0;  // this CTA's k-blocks (may be 0)

  if (threadIdx.x == 0) {
    for (int i = 0; i < C::kStages; ++i) {
      mbar_init(full(i), 1);
      mbar_init(empty(i), kConsumers);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  // first half of a cluster barrier: its wait, before the first store to another CTA's shared
  // memory, ensures every CTA of the cluster has started
  if (ck > 1) asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
  pdl_launch_dependents();
  pdl_wait();  // x is written by the preceding kernel, which may also still read u

  float d[4][NT][4];
#pragma unroll
  for (int mt = 0; mt < 4; ++mt)
#pragma unroll
    for (int t = 0; t < NT; ++t) d[mt][t][0] = d[mt][t][1] = d[mt][t][2] = d[mt][t][3] = 0.f;

  if (warp == kConsumers) {
    // ---------------------------------------------------------------- producer
    if (elect_one()) {
      tma_prefetch_desc(&tm_x);
      tma_prefetch_desc(&tm_a);
    }
    __syncwarp();
    int i = 0;
    for (; i < n; ++i) {
      const int st = i % C::kStages;
      if (i >= C::kStages && !warp_wait_bounded(empty(st), ((i / C::kStages) - 1) & 1, abort_flag, err,
                                             kDevTimeoutProducer))
        break;
      if (elect_one()) {
        const uint32_t dst = sbase + st * C::kStage;
        const int k = (kb0 + i) * 64;
        mbar_arrive_expect_tx(full(st), C::kStage);
        tma_load_2d(dst, &tm_x, k, row0, full(st));
        tma_load_2d(dst + kXTile, &tm_a, k, n_base, full(st));
      }
      __syncwarp();
    }
    // copies in flight land before the shared memory is reused or released
    volatile int no_abort = 0;
    for (int g = (i > C::kStages ? i - C::kStages : 0); g < i; ++g)
      warp_wait_bounded(full(g % C::kStages), (g / C::kStages) & 1, &no_abort, err, kDevTimeoutDrain);
  } else {
    // ---------------------------------------------------------------- consumers
    for (int i = 0; i < n; ++i) {
      const int st = i % C::kStages;
      if (!warp_wait_bounded(full(st), (i / C::kStages) & 1, abort_flag, err, kDevTimeoutEpilogue))
        break;
      const uint32_t xs = sbase + st * C::kStage;
      const uint32_t as = xs + kXTile;
      uint32_t a[4][4];
#pragma unroll
      for (int mt = 0; mt < 4; ++mt) {
        const int row = mt * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        ldsm_x4(xs + sw128(row, 2 * warp + (lane >> 4)), a[mt]);
      }
      if constexpr (NT == 1) {
        uint32_t b[2];
        const int nrow = lane & 7;
        ldsm_x2(as + sw128(nrow, 2 * warp + ((lane >> 3) & 1)), b);
#pragma unroll
        for (int mt = 0; mt < 4; ++mt) mma_bf16_16816(d[mt][0], a[mt], b[0], b[1]);
      } else {
#pragma unroll
        for (int tp = 0; tp < NT / 2; ++tp) {
          uint32_t b[4];
          const int nrow = 8 * (2 * tp + (lane >> 4)) + (lane & 7);
          ldsm_x4(as + sw128(nrow, 2 * warp + ((lane >> 3) & 1)), b);
#pragma unroll
          for (int mt = 0; mt < 4; ++mt) {
            mma_bf16_16816(d[mt][2 * tp], a[mt], b[0], b[1]);
            mma_bf16_16816(d[mt][2 * tp + 1], a[mt], b[2], b[3]);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(empty(st));
    }
  }
  __syncthreads();  // every stage is consumed and no copy is in flight: the ring is free

  // partial tiles of the consumer warps, summed in warp order
  float* part = reinterpret_cast<float*>(smem);
  float* recv = reinterpret_cast<float*>(smem + C::kRecvOff);
  if (warp < kConsumers) {
    float* pw = part + warp * (kBM * C::kLd);
    const int g = lane >> 2, c = lane & 3;
#pragma unroll
    for (int mt = 0; mt < 4; ++mt)
#pragma unroll
      for (int t = 0; t < NT; ++t) {
        *reinterpret_cast<float2*>(pw + (mt * 16 + g) * C::kLd + t * 8 + 2 * c) =
            make_float2(d[mt][t][0], d[mt][t][1]);
        *reinterpret_cast<float2*>(pw + (mt * 16 + g + 8) * C::kLd + t * 8 + 2 * c) =
            make_float2(d[mt][t][2], d[mt][t][3]);
      }
  }
  __syncthreads();
  if (ck > 1) asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
  const int rows_per = kBM / ck;
  constexpr int kQ = 2 * NT;  // float4 groups per row
  for (int e = threadIdx.x; e < kBM * kQ; e += kThreads) {
    const int rr = e / kQ, cc = (e % kQ) * 4;
    float4 v = *reinterpret_cast<const float4*>(part + rr * C::kLd + cc);
#pragma unroll
    for (int w = 1; w < kConsumers; ++w) {
      const float4 p = *reinterpret_cast<const float4*>(part + w * (kBM * C::kLd) + rr * C::kLd + cc);
      v.x += p.x;
      v.y += p.y;
      v.z += p.z;
      v.w += p.w;
    }
    if (ck > 1) {
      // row rr is finished by rank rr / rows_per, into its slot for this rank
      const int dst = rr / rows_per, lr = rr % rows_per;
      st_cluster_v4(recv + ((static_cast<int>(rank) * rows_per + lr) * 8 * NT + cc),
                    static_cast<uint32_t>(dst), v);
    } else {
      const int m = row0 + rr, nn = n_base + cc;
      if (m < M && nn < r) store_u4(u, r, m, nn, s, v);
    }
  }
  if (ck > 1) {
    cluster_sync_all();  // every CTA's pushes have landed and are visible
    for (int e = threadIdx.x; e < rows_per * kQ; e += kThreads) {
      const int lr = e / kQ, cc = (e % kQ) * 4;
      float4 v = *reinterpret_cast<const float4*>(recv + lr * 8 * NT + cc);
      for (int q = 1; q < ck; ++q) {
        const float4 p = *reinterpret_cast<const float4*>(recv + ((q * rows_per + lr) * 8 * NT + cc));
        v.x += p.x;
        v.y += p.y;
        v.z += p.z;
        v.w += p.w;
      }
      const int m = row0 + static_cast<int>(rank) * rows_per + lr, nn = n_base + cc;
      if (m < M && nn < r) store_u4(u, r, m, nn, s, v);
    }
  }
}

}  // namespace lds

// ---------------------------------------------------------------- dual_lora_gemv
//
// Decode-shaped dual-output linear (at most 16 token rows over both streams). HBM-bound:
// every byte of W is read once. One CTA per 16 rows of W; its warps (8, or 4 when there are
// at least four row blocks per SM) split K and stream their [16 x 64] W and token-row slices
// into XOR-swizzled shared memory with cp.async (3 stages per warp, 16-byte copies), then
// run mma.sync m16n8k16 with W as the 16-row operand and the token rows as the 8-wide
// operand (both through ldmatrix), so the arithmetic never limits the stream even at 16
// rows. The partial tiles are reduced in shared memory, where each thread also adds the
// rank-r LoRA term of its (row, token). (Measured on GB300: concurrent CTAs per SM matter
// more than ring depth; 4 warps per CTA lift the 11008- and 32000-row shapes by 10-25 %,
// while 4096-row shapes, 256 CTAs, need 8 warps to keep enough loads in flight.)

// per-warp ring: stage = 16 W rows + 8 NT token rows of 64 bf16, 3 stages
template <int NT, int W>  // NT n-tiles of 8 token rows, W warps
struct Gv {
  static constexpr int kStages = 3;
  static constexpr int kStageBytes = (16 + 8 * NT) * 128;
  static constexpr int kSmem = W * kStages * kStageBytes + W * 16 * 16 * 4;
};

__device__ __forceinline__ void gv_cp_async16(uint32_t dst, const void* src, bool ok) {
  const int n = ok ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n)
               : "memory");
}
__device__ __forceinline__ void gv_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void gv_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void gv_ldsm_x4(uint32_t addr, uint32_t (&a)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(a[0]), "=r"(a[1]), "=r"(a[2]), "=r"(a[3])
               : "r"(addr));
}

template <int NT, int kGvWarps, bool kAlias = false>  // kAlias: partial tiles in the ring
__global__ void __launch_bounds__(32 * kGvWarps)
    dual_lora_gemv_kernel(const __nv_bfloat16* __restrict__ x_off,
                          const __nv_bfloat16* __restrict__ x_on, int M, int K, int N,
                          const __nv_bfloat16* __restrict__ W, const __nv_bfloat16* __restrict__ u,
                          const __nv_bfloat16* __restrict__ B, int r, void* y_off, void* y_on,
                          int out_f32, int shared_x) {
  extern __shared__ __align__(1024) uint8_t smem[];
  constexpr int kGvStages = Gv<NT, kGvWarps>::kStages;
  constexpr int kGvStageBytes = Gv<NT, kGvWarps>::kStageBytes;
  float* red = reinterpret_cast<float*>(kAlias ? smem : smem + kGvWarps * kGvStages * kGvStageBytes);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int g = lane >> 2, c = lane & 3;
  const int n0 = blockIdx.x * 16;
  const int tokens = shared_x ? M : 2 * M;  // token rows: x_off rows, then x_on rows
  const uint32_t wsm = smem_u32(smem) + warp * kGvStages * kGvStageBytes;

  // this warp's K range in chunks of 64
  const int nchunk = (K + 63) / 64;
  const int per = (nchunk + kGvWarps - 1) / kGvWarps;
  const int c0 = warp * per;
  const int c1 = min(nchunk, c0 + per);

  // W is frozen: the first chunks of this warp's [16 x K-range] slice stream into L2 while
  // the preceding kernel finishes (programmatic dependent launch); x, u and y are touched
  // only after pdl_wait(). Prefetching the whole slice instead evicts, on the large
  // shapes, lines the running kernel has yet to read.
  pdl_launch_dependents();
  if (c0 < c1 && lane < 16 && n0 + lane < N)
    prefetch_l2_bulk(W + static_cast<size_t>(n0 + lane) * K + c0 * 64,
                     static_cast<uint32_t>(min(K, min(c1, c0 + kGvStages) * 64) - c0 * 64) * 2u);
  pdl_wait();

  // token row copied by this lane's slice of the x stage (rows lane >> 3 and 4 + lane >> 3...)
  auto xrow = [&](int tk) {
    return (tk < M) ? x_off + static_cast<size_t>(tk) * K : x_on + static_cast<size_t>(tk - M) * K;
  };
  auto issue = [&](int ch, int slot) {
    const uint32_t base = wsm + slot * kGvStageBytes;
    // W: 16 rows x 8 segments of 16 B, lane copies segments lane + 32 e
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int idx = lane + 32 * e;
      const int row = idx >> 3, seg = idx & 7;
      const int k = ch * 64 + seg * 8;
      const bool ok = (n0 + row < N) && (k < K);
      const __nv_bfloat16* src = W + static_cast<size_t>(ok ? n0 + row : 0) * K + (ok ? k : 0);
      gv_cp_async16(base + row * 128 + ((seg ^ (row & 7)) << 4), src, ok);
    }
    // token rows 0 .. 8 NT - 1 (missing rows and columns read as zero)
#pragma unroll
    for (int e = 0; e < NT * 2; ++e) {
      const int idx = lane + 32 * e;
      const int row = idx >> 3, seg = idx & 7;
      const int k = ch * 64 + seg * 8;
      const bool ok = (row < tokens) && (k < K);
      const __nv_bfloat16* src = ok ? xrow(row) + k : W;
      gv_cp_async16(base + 16 * 128 + row * 128 + ((seg ^ (row & 7)) << 4), src, ok);
    }
  };
  float d[NT][4];
#pragma unroll
  for (int t = 0; t < NT; ++t) d[t][0] = d[t][1] = d[t][2] = d[t][3] = 0.f;

  // prologue: up to kGvStages - 1 chunks in flight
#pragma unroll
  for (int i = 0; i < kGvStages - 1; ++i) {
    if (c0 + i < c1) issue(c0 + i, i);
    gv_commit();
  }
  for (int ch = c0; ch < c1; ++ch) {
    const int i = ch - c0;
    if (ch + kGvStages - 1 < c1) issue(ch + kGvStages - 1, (i + kGvStages - 1) % kGvStages);
    gv_commit();
    gv_wait<kGvStages - 1>();
    __syncwarp();
    const uint32_t st = wsm + (i % kGvStages) * kGvStageBytes;
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      const int k0 = ch * 64 + kk * 16;
      if (k0 >= K) break;
      uint32_t a[4];
      // matrices: rows (lane & 15), 16-byte segment 2 kk + (lane >> 4)
      const int row = lane & 15;
      gv_ldsm_x4(st + row * 128 + (((2 * kk + (lane >> 4)) ^ (row & 7)) << 4), a);
      // B fragments of token rows t*8 .. t*8 + 7: matrices (rows lane & 7, segment 2 kk and
      // 2 kk + 1) for n-tiles t = 0 (lanes 0-15) and t = 1 (lanes 16-31)
      uint32_t b[4];
      {
        const int trow = (lane & 7) + ((lane >> 4) << 3);
        const int seg = 2 * kk + ((lane >> 3) & 1);
        const uint32_t addr = st + 16 * 128 + trow * 128 + ((seg ^ (trow & 7)) << 4);
        if (NT == 2) {
          gv_ldsm_x4(addr, b);
        } else {  // token rows 0..7 only: two matrices, addresses from lanes 0-15
          asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0,%1}, [%2];"
                       : "=r"(b[0]), "=r"(b[1])
                       : "r"(addr));
        }
      }
#pragma unroll
      for (int t = 0; t < NT; ++t) mma_bf16_16816(d[t], a, b[2 * t], b[2 * t + 1]);
    }
    __syncwarp();
  }
  gv_wait<0>();
  if (kAlias) __syncthreads();  // the ring is free before it holds the partial tiles

  // partial [16 rows x 8 NT tokens] of this warp -> shared memory
  float* rw = red + warp * 16 * 16;
#pragma unroll
  for (int t = 0; t < NT; ++t) {
    rw[g * 16 + t * 8 + 2 * c] = d[t][0];
    rw[g * 16 + t * 8 + 2 * c + 1] = d[t][1];
    rw[(g + 8) * 16 + t * 8 + 2 * c] = d[t][2];
    rw[(g + 8) * 16 + t * 8 + 2 * c + 1] = d[t][3];
  }
  __syncthreads();
  // (row, token) outputs, row fastest for coalesced stores; 16 x 8 NT of them over the CTA
  for (int o = threadIdx.x; o < 16 * 8 * NT; o += 32 * kGvWarps) {
    const int row = o & 15, tk = o >> 4;
    const int n = n0 + row;
    if (tk >= tokens || n >= N) continue;
    float acc = 0.f;
#pragma unroll
    for (int w = 0; w < kGvWarps; ++w) acc += red[w * 256 + row * 16 + tk];
    auto put = [&](void* y, int m, float v) {
      if (y == nullptr) return;
      const size_t off = static_cast<size_t>(m) * N + n;
      if (out_f32)
        reinterpret_cast<float*>(y)[off] = v;
      else
        reinterpret_cast<__nv_bfloat16*>(y)[off] = __float2bfloat16_rn(v);
    };
    auto lora = [&](int m) {
      // rank-r dot product with 16-byte loads (r % 8 == 0)
      float v = 0.f;
      if (u != nullptr) {
        const uint4* up = reinterpret_cast<const uint4*>(u + static_cast<size_t>(m) * r);
        const uint4* bp = reinterpret_cast<const uint4*>(B + static_cast<size_t>(n) * r);
        for (int j = 0; j < r / 8; ++j) {
          const uint4 a4 = __ldg(up + j), b4 = __ldg(bp + j);
          const uint32_t* ap = &a4.x;
          const uint32_t* bq = &b4.x;
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 fa = unpack_bf16x2(ap[e]), fb = unpack_bf16x2(bq[e]);
            v = fmaf(fa.x, fb.x, v);
            v = fmaf(fa.y, fb.y, v);
          }
        }
      }
      return v;
    };
    if (shared_x) {
      put(y_off, tk, acc);
      if (y_on != nullptr) put(y_on, tk, acc + lora(tk));
    } else if (tk < M) {
      put(y_off, tk, acc);
    } else {
      put(y_on, tk - M, acc + lora(tk - M));
    }
  }
}

template <int NT, int W>
void launch_gemv_t(const GemmArgs& a, int nsm, cudaStream_t stream) {
  constexpr int smem_full = Gv<NT, W>::kSmem;
  constexpr int smem_ring = W * Gv<NT, W>::kStages * Gv<NT, W>::kStageBytes;
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(dual_lora_gemv_kernel<NT, W>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         smem_full);
    cudaFuncSetAttribute(dual_lora_gemv_kernel<NT, W, true>,
                         cudaFuncAttributeMaxDynamicSharedMemorySize, smem_ring);
    attr = true;
  }
  const unsigned grid = static_cast<unsigned>((a.N + 15) / 16);
  // the partial tiles in the ring, one more CTA per SM, only where that brings a grid that
  // just misses one wave into one (the 768-CTA q/k/v shape against 5 x 152 = 760 slots)
  const int per_sm = 227 * 1024 / (smem_full + 1024);
  const int per_sm_alias = 227 * 1024 / (smem_ring + 1024);
  const bool alias = per_sm_alias > per_sm && static_cast<int>(grid) > per_sm * nsm &&
                     static_cast<int>(grid) <= per_sm_alias * nsm;
  const int smem = alias ? smem_ring : smem_full;
  launch_pdl(alias ? dual_lora_gemv_kernel<NT, W, true> : dual_lora_gemv_kernel<NT, W>,
      dim3(grid), dim3(32 * W), smem, stream,
      static_cast<const __nv_bfloat16*>(a.x_off),
      static_cast<const __nv_bfloat16*>(a.shared_x ? a.x_off : a.x_on), static_cast<int>(a.M),
      static_cast<int>(a.K), static_cast<int>(a.N), static_cast<const __nv_bfloat16*>(a.W),
      static_cast<const __nv_bfloat16*>(a.u), static_cast<const __nv_bfloat16*>(a.B),
      static_cast<int>(a.r), a.y_off, a.y_on, a.out_f32, a.shared_x ? 1 : 0);
}

// Streaming lora_down: clusters of ck CTAs (a power of two up to 8) along K, ck as large as
// still lets every CTA of the launch be resident at once, and at least one k-block per CTA.
template <int NT>
int launch_lora_down_stream(const void* x, int64_t M, int64_t K, const void* A, int64_t r,
                            float s, void* u, int nsm, cudaStream_t stream) {
  using C = lds::Cfg<NT>;
  static bool attr = false;
  if (!attr) {
    if (cudaFuncSetAttribute(lds::lora_down_stream_kernel<NT>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem) != cudaSuccess)
      return -1;
    attr = true;
  }
  int* err = device_error_word();
  if (err == nullptr) return -1;
  CUtensorMap mx, ma;
  if (!make_tma_map(&mx, x, M, K, K, lds::kBM, false)) return -2;
  if (!make_tma_map(&ma, A, r, K, K, 8 * NT, false)) return -2;
  const int64_t rb = (M + lds::kBM - 1) / lds::kBM;
  const int64_t ny = (r + 63) / 64;
  const int64_t per_sm = std::max<int64_t>(1, (227 * 1024) / C::kSmem);
  const int64_t fit = std::max<int64_t>(1, per_sm * nsm / (rb * ny));
  const int64_t nkb = (K + 63) / 64;
  int ck = 1;
  while (ck < 8 && 2 * ck <= fit && 2 * ck <= nkb) ck *= 2;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(rb * ck), static_cast<unsigned>(ny));
  cfg.blockDim = dim3(lds::kThreads);
  cfg.dynamicSmemBytes = C::kSmem;
  cfg.stream = stream;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  at[1].id = cudaLaunchAttributeClusterDimension;
  at[1].val.clusterDim.x = static_cast<unsigned>(ck);
  at[1].val.clusterDim.y = 1;
  at[1].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = ck > 1 ? 2 : 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, lds::lora_down_stream_kernel<NT>, mx, ma,
                                           static_cast<int>(M), static_cast<int>(K),
                                           static_cast<int>(r), s, static_cast<__nv_bfloat16*>(u),
                                           ck, err);
  return e == cudaSuccess ? 0 : -3;
}

}  // namespace

int launch_lora_down(const void* x, int64_t M, int64_t K, const void* A, int64_t r, float s,
                     void* u, cudaStream_t stream) {
  if (M == 0 || r == 0) return 0;
  static int nsm = 0;
  if (nsm == 0) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return -1;
  }
  const auto* xp = static_cast<const __nv_bfloat16*>(x);
  const auto* ap = static_cast<const __nv_bfloat16*>(A);
  auto* up = static_cast<__nv_bfloat16*>(u);
  if (M >= lds::kBM && K >= 64) {
    if (r <= 8) return launch_lora_down_stream<1>(x, M, K, A, r, s, u, nsm, stream);
    if (r <= 16) return launch_lora_down_stream<2>(x, M, K, A, r, s, u, nsm, stream);
    if (r <= 32) return launch_lora_down_stream<4>(x, M, K, A, r, s, u, nsm, stream);
    return launch_lora_down_stream<8>(x, M, K, A, r, s, u, nsm, stream);
  }
  const int64_t tiles = (M + 15) / 16;
  const int64_t ny = r <= 32 ? 1 : (r + 63) / 64;
  // K split over a cluster: about 4 CTAs per SM (2 above 16 ranks, where each CTA already
  // reads more of A than of x), each warp with at least 4 chunks of 32 (one unrolled batch of
  // loads)
  const int64_t target = (r > 16 ? 2LL : 4LL) * nsm;
  int64_t ck = (target + tiles * ny - 1) / (tiles * ny);
  ck = std::min<int64_t>(ck, std::max<int64_t>(1, K / (32 * 4 * kDownWarps)));
  ck = std::max<int64_t>(1, std::min<int64_t>(8, ck));
  const dim3 grid(static_cast<unsigned>(tiles * ck), static_cast<unsigned>(ny));
  const int Mi = static_cast<int>(M), Ki = static_cast<int>(K), ri = static_cast<int>(r);
  const int cki = static_cast<int>(ck);
  cudaError_t e;
  if (r <= 8)
    e = launch_down(lora_down_kernel<1>, grid, cki, stream, xp, Mi, Ki, ap, ri, s, up, cki);
  else if (r <= 16)
    e = launch_down(lora_down_kernel<2>, grid, cki, stream, xp, Mi, Ki, ap, ri, s, up, cki);
  else if (r <= 32)
    e = launch_down(lora_down_kernel<4>, grid, cki, stream, xp, Mi, Ki, ap, ri, s, up, cki);
  else
    e = launch_down(lora_down_kernel<8>, grid, cki, stream, xp, Mi, Ki, ap, ri, s, up, cki);
  return e == cudaSuccess ? 0 : -3;
}

int launch_dual_lora_gemv(const GemmArgs& a, cudaStream_t stream) {
  const int64_t rows = a.shared_x ? a.M : 2 * a.M;
  int dev = 0, nsm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return -1;
  const bool narrow = (a.N + 15) / 16 >= 4LL * nsm;  // enough row blocks for 4-warp CTAs
  if (rows <= 8) {
    if (narrow)
      launch_gemv_t<1, 4>(a, nsm, stream);
    else
      launch_gemv_t<1, 8>(a, nsm, stream);
  } else {
    if (narrow)
      launch_gemv_t<2, 4>(a, nsm, stream);
    else
      launch_gemv_t<2, 8>(a, nsm, stream);
  }
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace hydra
