// Skinny dual-stream LoRA linear for decode-sized batches (tcgen05, split-K over a cluster).
//
// A decode step multiplies at most 128 token rows (the LoRA-off rows of every sequence,
// then the LoRA-on rows) by each frozen weight W [N, K]. The work is reading W once
// (§3 Dynamic LoRA: one frozen W serves both streams). With one 128 x bn tile per CTA and
// K whole in each CTA, a 4096-wide projection has 16 tiles: 16 SMs stream W and HBM stays
// mostly idle. Here the K range of each tile is split over a thread-block cluster of ks
// CTAs (ks <= 8): every CTA streams W[n0 : n0 + bn, its K slice] through a TMA ring into
// tcgen05 MMAs with the 128 rows of x as the A operand, so tiles x ks CTAs stream W.
//
// Both streams share one A tile: rows [0, u_row0) are the off rows and take x W^T; rows
// [u_row0, u_row0 + M_u) also take the LoRA term u B^T (u = s x_on A^T, computed before).
// The LoRA k-blocks load u at row coordinate -u_row0, so TMA fills the off rows of that
// operand with zeros and the one MMA stream adds exactly 0 to them.
//
// Reduction: every CTA finishes its partial sum in TMEM. Each rank owns a slice of the
// tile's columns. It writes the other ranks' slices of its partial to its shared memory
// as fp32, and after a cluster barrier sums its own slice over the ranks in rank order
// (partials of the other ranks read through distributed shared memory). The order is
// fixed, so results are deterministic; it is a different association of the same fp32
// dot product than a single-CTA pass. Output: y [M, N] row-major, bf16 (rounded once
// from the fp32 sum) or fp32.
//
// Roles per CTA (192 threads): warp 0 TMA producer, warp 1 MMA issuer (TMEM allocation),
// warps 2-5 epilogue (TMEM lanes 32 (w % 4) .. + 31). Every mbarrier wait is bounded; on
// expiry the CTA records an error, skips its remaining work and still reaches both
// cluster barriers, so no CTA of the cluster waits on it forever.
#include "common.cuh"
#include "kernels.h"

#include <mutex>
#include <vector>

namespace hydra {
namespace skinny {

constexpr int BM = 128;
constexpr int BK = 64;
constexpr int A_TILE = BM * BK * 2;  // 16 KiB
constexpr int NUM_THREADS = 192;
constexpr int kMaxStages = 12;
constexpr int kMaxBN = 256;
constexpr int kMaxKs = 8;
constexpr uint32_t kTmemCols = 256;
constexpr int kSmemMax = 232448;  // dynamic shared memory limit of one CTA (227 KiB)
constexpr int kSmemTail = 1024 + (2 * kMaxStages + 1) * 8 + 16;  // alignment pad, barriers

struct Params {
  int M, N;
  int kb_main;  // ceil(K / BK)
  int kb_lora;  // ceil(r / BK); 0 = no LoRA
  int r;
  int u_row0;   // first row of the tile that takes the LoRA term
  int bn, ks, stages, stage_bytes;
  uint32_t idesc;
  int out_f32;
  void* y;
  int* err;
};

__device__ __forceinline__ float4 ld_cluster_v4(uint32_t cluster_addr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(cluster_addr)
               : "memory");
  return v;
}

__device__ __forceinline__ void st_shared_f4(uint32_t addr, float a, float b, float c, float d) {
  asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(a), "f"(b), "f"(c),
               "f"(d)
               : "memory");
}

// 16 consecutive columns of one output row (16 columns never straddle N: N % 16 == 0)
__device__ __forceinline__ void store16(const Params& p, int row, int col, const float (&v)[16]) {
  if (p.out_f32) {
    float4* d = reinterpret_cast<float4*>(static_cast<float*>(p.y) + static_cast<size_t>(row) * p.N + col);
#pragma unroll
    for (int j = 0; j < 4; ++j) d[j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
  } else {
    uint4* d = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(p.y) + static_cast<size_t>(row) * p.N + col);
#pragma unroll
    for (int j = 0; j < 2; ++j)
      d[j] = make_uint4(pack_bf16x2(v[8 * j], v[8 * j + 1]), pack_bf16x2(v[8 * j + 2], v[8 * j + 3]),
                        pack_bf16x2(v[8 * j + 4], v[8 * j + 5]), pack_bf16x2(v[8 * j + 6], v[8 * j + 7]));
  }
}

__global__ void __launch_bounds__(NUM_THREADS, 1)
    skinny_gemm_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_w,
                       const __grid_constant__ CUtensorMap tm_u, const __grid_constant__ CUtensorMap tm_b,
                       const Params p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + p.stages * p.stage_bytes);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kMaxStages + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int ks = p.ks;
  const int rank = ks > 1 ? static_cast<int>(cluster_rank()) : 0;
  const int n0 = static_cast<int>(blockIdx.x / ks) * p.bn;
  // this rank's k-blocks; the LoRA k-blocks go to the last rank
  const int kb0 = rank * p.kb_main / ks;
  const int kb1 = (rank + 1) * p.kb_main / ks;
  const int n_main = kb1 - kb0;
  const int items = n_main + (rank == ks - 1 ? p.kb_lora : 0);

  const uint32_t smem_base = smem_u32(smem);
  auto full_bar = [&](int s) { return smem_u32(&bars[s]); };
  auto empty_bar = [&](int s) { return smem_u32(&bars[kMaxStages + s]); };
  const uint32_t acc_full = smem_u32(&bars[2 * kMaxStages]);

  if (threadIdx.x == 0) {
    for (int s = 0; s < p.stages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(acc_full, 1);
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
  const uint32_t tmem_acc = *tmem_slot;

  bool epi_ok = false;
  if (warp == 0) {
    // ------------------------------------------------------------------ TMA producer
    if (elect_one()) {
      tma_prefetch_desc(&tm_x);
      tma_prefetch_desc(&tm_w);
      if (p.kb_lora > 0) {
        tma_prefetch_desc(&tm_u);
        tma_prefetch_desc(&tm_b);
      }
    }
    __syncwarp();
    // Programmatic dependent launch: W and B are frozen, so the weight halves of the first
    // ring's worth of items load before the wait on the preceding kernel (which writes x and
    // u); a stage's barrier completes only once its x half, loaded after the wait, lands too.
    const int pre = min(items, p.stages);
    if (elect_one()) {
      for (int i = 0; i < pre; ++i) {
        mbar_arrive_expect_tx(full_bar(i), p.stage_bytes);
        const uint32_t b_dst = smem_base + i * p.stage_bytes + A_TILE;
        if (i < n_main) tma_load_2d(b_dst, &tm_w, (kb0 + i) * BK, n0, full_bar(i));
        else tma_load_2d(b_dst, &tm_b, (i - n_main) * BK, n0, full_bar(i));
      }
    }
    __syncwarp();
    pdl_wait();
    int it = 0;
    for (; it < items; ++it) {
      const int s = it % p.stages;
      if (!warp_wait_bounded(empty_bar(s), ((it / p.stages) & 1) ^ 1, abort_flag, p.err,
                             kDevTimeoutProducer))
        break;
      if (elect_one()) {
        if (it >= pre) mbar_arrive_expect_tx(full_bar(s), p.stage_bytes);
        const uint32_t a_dst = smem_base + s * p.stage_bytes;
        if (it < n_main) {
          const int k = (kb0 + it) * BK;
          tma_load_2d(a_dst, &tm_x, k, 0, full_bar(s));
          if (it >= pre) tma_load_2d(a_dst + A_TILE, &tm_w, k, n0, full_bar(s));
        } else {
          const int k = (it - n_main) * BK;
          tma_load_2d(a_dst, &tm_u, k, -p.u_row0, full_bar(s));  // rows above u_row0: zeros
          if (it >= pre) tma_load_2d(a_dst + A_TILE, &tm_b, k, n0, full_bar(s));
        }
      }
      __syncwarp();
    }
    // copies still in flight land before shared memory is reused or released
    for (int k = (it > p.stages ? it - p.stages : 0); k < it; ++k) {
      volatile int no_abort = 0;
      warp_wait_bounded(full_bar(k % p.stages), (k / p.stages) & 1, &no_abort, p.err, kDevTimeoutDrain);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer
    for (int it = 0; it < items; ++it) {
      const int s = it % p.stages;
      if (!warp_wait_bounded(full_bar(s), (it / p.stages) & 1, abort_flag, p.err, kDevTimeoutMma))
        break;
      tc_fence_after();
      if (elect_one()) {
        const uint32_t a_base = smem_base + s * p.stage_bytes;
        const uint32_t b_base = a_base + A_TILE;
        const int nsub = it < n_main ? BK / 16 : min(BK / 16, (p.r - (it - n_main) * BK + 15) / 16);
        for (int k = 0; k < nsub; ++k)
          tc_mma_bf16(tmem_acc, smem_desc_sw128(a_base + k * 32), smem_desc_sw128(b_base + k * 32),
                      p.idesc, (it > 0 || k > 0) ? 1u : 0u);
        tc_commit(empty_bar(s));
      }
      __syncwarp();
    }
    // arrives once every MMA issued above is done (also after an abort, so TMEM is idle
    // before it is released)
    if (elect_one()) tc_commit(acc_full);
    __syncwarp();
    volatile int no_abort = 0;
    warp_wait_bounded(acc_full, 0, &no_abort, p.err, kDevTimeoutDrain);
  } else {
    // ------------------------------------------------------------------ epilogue
    epi_ok = mbar_wait_bounded(acc_full, 0, abort_flag, p.err, kDevTimeoutEpilogue);
    epi_ok = __all_sync(0xffffffffu, epi_ok) && *abort_flag == 0;
    tc_fence_after();
  }

  const int q = warp & 3;  // TMEM lanes of an epilogue warp
  const int row = q * 32 + lane;
  const uint32_t lane_taddr = tmem_acc + (static_cast<uint32_t>(q * 32) << 16);
  const bool warp_rows = q * 32 < p.M;  // warp-uniform: the warp holds at least one output row
  const int cols = min(p.bn, p.N - n0);   // valid columns of this tile (a multiple of 16)

  if (ks == 1) {
    if (warp >= 2 && epi_ok && warp_rows) {
      for (int c = 0; c < cols; c += 16) {
        uint32_t v[16];
        tc_ld_32x32b_x16(lane_taddr + c, v);
        tc_wait_ld();
        float f[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) f[i] = __uint_as_float(v[i]);
        if (row < p.M) store16(p, row, n0 + c, f);
      }
    }
  } else {
    // this rank's column slice [c_lo, c_hi) of the tile, 16-column granular
    const int cw = ((p.bn / ks) + 15) / 16 * 16;
    const int c_lo = min(cols, rank * cw);
    const int c_hi = min(cols, c_lo + cw);
    // exchange layout over the (now idle) ring: fp32 partial (row, col) at float4 index
    // (col / 4) * 128 + row, so a warp's 32 rows of one float4 column are contiguous
    const uint32_t xch = smem_base;
    if (warp >= 2 && epi_ok && warp_rows) {
      for (int c = 0; c < cols; c += 16) {
        if (c >= c_lo && c < c_hi) continue;
        uint32_t v[16];
        tc_ld_32x32b_x16(lane_taddr + c, v);
        tc_wait_ld();
#pragma unroll
        for (int j = 0; j < 4; ++j)
          st_shared_f4(xch + ((c / 4 + j) * BM + row) * 16, __uint_as_float(v[4 * j]),
                       __uint_as_float(v[4 * j + 1]), __uint_as_float(v[4 * j + 2]),
                       __uint_as_float(v[4 * j + 3]));
      }
    }
    tc_fence_before();
    cluster_sync_all();  // every rank's partials are in its shared memory
    if (warp >= 2 && epi_ok && warp_rows) {
      for (int c = c_lo; c < c_hi; c += 16) {
        uint32_t own[16];
        tc_ld_32x32b_x16(lane_taddr + c, own);
        tc_wait_ld();
        float f[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) f[i] = 0.f;
        for (int rr = 0; rr < ks; ++rr) {  // fixed association: ((p_0 + p_1) + p_2) + ...
          if (rr == rank) {
#pragma unroll
            for (int i = 0; i < 16; ++i) f[i] += __uint_as_float(own[i]);
          } else {
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const float4 t = ld_cluster_v4(map_to_rank(xch + ((c / 4 + j) * BM + row) * 16, rr));
              f[4 * j] += t.x;
              f[4 * j + 1] += t.y;
              f[4 * j + 2] += t.z;
              f[4 * j + 3] += t.w;
            }
          }
        }
        if (row < p.M) store16(p, row, n0 + c, f);
      }
    }
    cluster_sync_all();  // no rank leaves while another still reads its partials
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_acc, kTmemCols);
  }
}

}  // namespace skinny

// ------------------------------------------------------------------ host side

namespace {

struct Choice {
  int bn, ks, stages;
};

int stages_for(int bn) {
  const int stage = skinny::A_TILE + bn * 128;
  int s = (skinny::kSmemMax - skinny::kSmemTail) / stage;
  return s > skinny::kMaxStages ? skinny::kMaxStages : s;
}

size_t smem_bytes(int bn, int stages) {
  return static_cast<size_t>(stages) * (skinny::A_TILE + bn * 128) + skinny::kSmemTail;
}

// Clusters of ks CTAs with this shared-memory size that fit on the device at once.
int active_clusters(int dev, int ks, size_t smem) {
  static std::mutex mu;
  static std::vector<std::pair<long long, int>> cache;
  const long long key = static_cast<long long>(dev) << 48 | static_cast<long long>(ks) << 32 |
                        static_cast<long long>(smem);
  std::lock_guard<std::mutex> lock(mu);
  for (auto& e : cache)
    if (e.first == key) return e.second;
  int nsm = 0;
  if (cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  int n = nsm / ks;
  if (ks > 1) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(ks * (nsm / ks)));
    cfg.blockDim = dim3(skinny::NUM_THREADS);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = static_cast<unsigned>(ks);
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int c = 0;
    if (cudaOccupancyMaxActiveClusters(&c, skinny::skinny_gemm_kernel, &cfg) != cudaSuccess) {
      cudaGetLastError();
      c = 0;
    }
    n = c;
  }
  cache.emplace_back(key, n);
  return n;
}

// Tile width and cluster size by a cost model of the kernel (microseconds), fitted on
// GB300 to a sweep of the decode shapes (a pick within 4 % of the best measured one):
//  * an SM takes about 100 GB/s of TMA loads; a k-block costs a CTA its full 128-row x
//    tile (rows past M are filled with zeros but still cost) plus bn rows of W, 128 B each;
//  * all of W crosses HBM once, at about 6.5 TB/s;
//  * every wave of CTAs pays about 4 us of launch, set-up, pipeline fill and stores;
//  * a cluster adds about 1 us of barriers plus the exchange: ks - 1 partial slices of
//    M x (bn / ks) fp32 read through distributed shared memory at about 120 GB/s.
// Clusters beyond what fits on the device at once run in further waves.
Choice choose(int dev, int64_t M, int64_t K, int64_t N, int64_t r) {
  const int64_t kb = (K + skinny::BK - 1) / skinny::BK;
  const double t_hbm = 2.0 * static_cast<double>(N) * static_cast<double>(K + r) / 6.5e6;
  Choice best{256, 1, stages_for(256)};
  double best_t = 1e30;
  for (int bn : {256, 224, 192, 160, 128, 96, 64}) {
    const int stages = stages_for(bn);
    const int64_t tiles = (N + bn - 1) / bn;
    for (int ks = 1; ks <= skinny::kMaxKs; ++ks) {
      if (ks > kb) break;
      const int cw = ((bn / ks) + 15) / 16 * 16;
      if (ks > 1 && static_cast<int64_t>(cw) * (ks - 1) >= bn) continue;  // a rank with no columns
      const int fit = active_clusters(dev, ks, smem_bytes(bn, stages));
      if (fit < 1) continue;
      const double waves = static_cast<double>((tiles + fit - 1) / fit);
      const double kb_cta = static_cast<double>((kb + ks - 1) / ks);
      const double t_cta = kb_cta * (skinny::BM + bn) * 128.0 / 100000.0;
      const double xch =
          ks == 1 ? 0.0 : 1.0 + (ks - 1) * static_cast<double>(M) * cw * 4.0 / 120000.0;
      double t = waves * (t_cta + xch + 4.0);
      if (t < t_hbm + xch + 4.0) t = t_hbm + xch + 4.0;
      if (t < best_t * 0.999) {
        best_t = t;
        best = Choice{bn, ks, stages};
      }
    }
  }
  return best;
}

Choice cached_choice(int dev, int64_t M, int64_t K, int64_t N, int64_t r) {
  struct Entry {
    int dev;
    int64_t M, K, N, r;
    Choice c;
  };
  static std::mutex mu;
  static std::vector<Entry> cache;
  {
    std::lock_guard<std::mutex> lock(mu);
    for (auto& e : cache)
      if (e.dev == dev && e.M == M && e.K == K && e.N == N && e.r == r) return e.c;
  }
  const Choice c = choose(dev, M, K, N, r);
  std::lock_guard<std::mutex> lock(mu);
  if (cache.size() < 256) cache.push_back(Entry{dev, M, K, N, r, c});
  return c;
}

}  // namespace

bool skinny_gemm_supported(int64_t M, int64_t K, int64_t N, int64_t r) {
  return M >= 1 && M <= skinny::BM && K >= 1 && K % 8 == 0 && N >= 16 && N % 16 == 0 &&
         r >= 0 && r % 8 == 0 && N <= (int64_t{1} << 30) && K <= (int64_t{1} << 30);
}

int launch_skinny_gemm_tc(const SkinnyArgs& a, cudaStream_t st) {
  using namespace skinny;
  if (!skinny_gemm_supported(a.M, a.K, a.N, a.r)) return -4;
  if (a.r > 0 && (a.u == nullptr || a.B == nullptr || a.u_rows < 1 || a.u_row0 < 0 ||
                  a.u_row0 + a.u_rows > a.M))
    return -4;
  // the shared-memory limit is a per-device function attribute: set once per device
  static bool attr_set[64] = {false};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return -1;
  if (!attr_set[dev]) {
    if (cudaFuncSetAttribute(skinny_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kSmemMax) != cudaSuccess)
      return -1;
    attr_set[dev] = true;
  }
  Choice c = cached_choice(dev, a.M, a.K, a.N, a.r);
  if (a.bn > 0) {  // explicit tile width / cluster size (sweeps and tests)
    if (a.bn % 16 != 0 || a.bn > kMaxBN) return -4;
    c.bn = a.bn;
    c.stages = stages_for(a.bn);
  }
  if (a.ks > 0) {
    const int64_t kb = (a.K + BK - 1) / BK;
    if (a.ks > kMaxKs || a.ks > kb) return -4;
    c.ks = a.ks;
  }
  if (c.stages < 2) return -4;
  const int64_t tiles = (a.N + c.bn - 1) / c.bn;

  CUtensorMap mx, mw, mu, mb;
  if (!make_tma_map(&mx, a.x, a.M, a.K, a.K, BM, false)) return -2;
  if (!make_tma_map(&mw, a.W, a.N, a.K, a.K, c.bn, false)) return -2;
  if (a.r > 0) {
    if (!make_tma_map(&mu, a.u, a.u_rows, a.r, a.r, BM, false)) return -2;
    if (!make_tma_map(&mb, a.B, a.N, a.r, a.r, c.bn, false)) return -2;
  } else {  // never read
    mu = mx;
    mb = mw;
  }
  Params p;
  p.M = static_cast<int>(a.M);
  p.N = static_cast<int>(a.N);
  p.kb_main = static_cast<int>((a.K + BK - 1) / BK);
  p.kb_lora = a.r > 0 ? static_cast<int>((a.r + BK - 1) / BK) : 0;
  p.r = static_cast<int>(a.r);
  p.u_row0 = static_cast<int>(a.u_row0);
  p.bn = c.bn;
  p.ks = c.ks;
  p.stages = c.stages;
  p.stage_bytes = A_TILE + c.bn * 128;
  p.idesc = idesc_bf16_f32(BM, c.bn);
  p.out_f32 = a.out_f32;
  p.y = a.y;
  p.err = a.err;

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(tiles * c.ks));
  cfg.blockDim = dim3(NUM_THREADS);
  cfg.dynamicSmemBytes = smem_bytes(c.bn, c.stages);
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(c.ks);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, skinny_gemm_kernel, mx, mw, mu, mb, p) == cudaSuccess ? 0 : -3;
}

}  // namespace hydra
