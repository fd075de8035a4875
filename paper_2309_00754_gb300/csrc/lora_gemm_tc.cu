// Dual-output LoRA linear on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
// One frozen weight W serves both roles of the Hydra model (§3 Dynamic LoRA: the
// reference policy is the actor with its LoRA parameters ignored):
//     y_off = x_off W^T                 (LoRA off: reference / reward stream)
//     y_on  = x_on  W^T + u B^T,  u = s x_on A^T   (LoRA on: actor / critic stream)
// Storage: x [M, K], W [N, K], u [M, r], B [N, r], all bf16 row-major (K-major operands).
//
// Two tile kinds share one kernel:
//  * shared input (x_on == x_off): the tile's x W^T accumulates once in TMEM; the
//    epilogue drains it to y_off, then the MMA thread accumulates u B^T on top of the same
//    TMEM accumulator and the epilogue drains y_on. One read of each W tile yields both.
//  * stacked streams (x_on != x_off): tiles of the off stream produce y_off; tiles of the on
//    stream run the main loop followed by the LoRA k-blocks ([x_on | u] [W | B]^T) into one
//    accumulator and produce y_on. Off and on tiles of the same n-block run next to each
//    other, so each W tile is fetched from HBM once and re-read from L2.
//
// CTA layout (192 threads): warp 0 = TMA producer, warp 1 = TMEM owner + MMA issuer,
// warps 2..5 = epilogue (warp w reads TMEM lanes 32*(w%4) .. +31).
// Tile 128 x 256 x 64, 4-stage shared-memory ring, bf16 inputs, fp32 accumulation,
// 128-byte-swizzled K-major operands.
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
constexpr uint32_t TMEM_COLS = 256;
constexpr int NUM_BARS = 2 * STAGES + 3;
constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + NUM_BARS * 8 + 64;
constexpr uint32_t IDESC = idesc_bf16_f32(BM, BN);

struct Params {
  int M, N, K;
  int kb_main;   // ceil(K / BK)
  int kb_lora;   // ceil(r / BK); 0 = no LoRA
  int r;
  int shared_x;  // 1 = x_on is x_off
  int m_tiles, n_tiles;
  void* y_off;
  void* y_on;
  int out_f32;
  int* err;
};

__device__ __forceinline__ void store_chunk(void* y, int out_f32, int N, int m, int n,
                                            const uint32_t (&v)[32]) {
  if (out_f32) {
    float* row = reinterpret_cast<float*>(y) + static_cast<size_t>(m) * N + n;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (n + 4 * j < N) {
        float4 f = make_float4(__uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]),
                               __uint_as_float(v[4 * j + 2]), __uint_as_float(v[4 * j + 3]));
        *reinterpret_cast<float4*>(row + 4 * j) = f;
      }
    }
  } else {
    __nv_bfloat16* row = reinterpret_cast<__nv_bfloat16*>(y) + static_cast<size_t>(m) * N + n;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (n + 8 * j < N) {
        uint4 q;
        q.x = pack_bf16x2(__uint_as_float(v[8 * j + 0]), __uint_as_float(v[8 * j + 1]));
        q.y = pack_bf16x2(__uint_as_float(v[8 * j + 2]), __uint_as_float(v[8 * j + 3]));
        q.z = pack_bf16x2(__uint_as_float(v[8 * j + 4]), __uint_as_float(v[8 * j + 5]));
        q.w = pack_bf16x2(__uint_as_float(v[8 * j + 6]), __uint_as_float(v[8 * j + 7]));
        *reinterpret_cast<uint4*>(row + 8 * j) = q;
      }
    }
  }
}

// Epilogue warp: read the 32 TMEM lanes of this warp (tile rows) across the tile's columns
// and store them to up to two outputs.
__device__ __forceinline__ void drain(uint32_t tmem_row, int m, int M, int n0, const Params& p,
                                      void* t0, void* t1) {
#pragma unroll 1
  for (int c = 0; c < BN / 32; ++c) {
    uint32_t v[32];
    tc_ld_32x32b_x32(tmem_row + c * 32, v);
    tc_wait_ld();
    const int n = n0 + c * 32;
    if (m < M && n < p.N) {
      if (t0) store_chunk(t0, p.out_f32, p.N, m, n, v);
      if (t1) store_chunk(t1, p.out_f32, p.N, m, n, v);
    }
  }
}

__global__ void __launch_bounds__(NUM_THREADS, 1)
    dual_lora_gemm_kernel(const __grid_constant__ CUtensorMap tm_x_off,
                          const __grid_constant__ CUtensorMap tm_x_on,
                          const __grid_constant__ CUtensorMap tm_w,
                          const __grid_constant__ CUtensorMap tm_u,
                          const __grid_constant__ CUtensorMap tm_b, const Params p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + NUM_BARS);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  // tile -> (stream, m-block, n-block); off/on tiles of one (m, n) are adjacent
  const int streams = p.shared_x ? 1 : 2;
  int t = blockIdx.x;
  const int stream = t % streams;
  t /= streams;
  const int m_idx = t % p.m_tiles;
  const int n_idx = t / p.m_tiles;
  const int m0 = m_idx * BM;
  const int n0 = n_idx * BN;

  const bool on_stream = p.shared_x ? true : (stream == 1);
  const int n_lora = (p.kb_lora > 0 && on_stream && p.y_on != nullptr) ? p.kb_lora : 0;
  const bool mid_drain = p.shared_x && n_lora > 0 && p.y_off != nullptr;
  const int total_kb = p.kb_main + n_lora;
  const CUtensorMap* tmx = (stream == 1) ? &tm_x_on : &tm_x_off;

  // final drain targets
  void* fin0;
  void* fin1 = nullptr;
  if (p.shared_x) {
    if (n_lora > 0) {
      fin0 = p.y_on;
    } else {
      fin0 = p.y_off;
      fin1 = p.y_on;
    }
  } else {
    fin0 = (stream == 1) ? p.y_on : p.y_off;
  }

  const uint32_t smem_base = smem_u32(smem);
  auto full_bar = [&](int s) { return smem_u32(&bars[s]); };
  auto empty_bar = [&](int s) { return smem_u32(&bars[STAGES + s]); };
  const uint32_t acc_full = smem_u32(&bars[2 * STAGES]);
  const uint32_t acc_empty = smem_u32(&bars[2 * STAGES + 1]);
  const uint32_t mma_done = smem_u32(&bars[2 * STAGES + 2]);

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, 128);
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tm_x_off);
    tma_prefetch_desc(&tm_x_on);
    tma_prefetch_desc(&tm_w);
    tma_prefetch_desc(&tm_u);
    tma_prefetch_desc(&tm_b);
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
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer
      int issued = 0;
      for (int kb = 0; kb < total_kb; ++kb) {
        const int s = kb % STAGES;
        const uint32_t ph = (kb / STAGES) & 1;
        if (!mbar_wait_bounded(empty_bar(s), ph ^ 1, abort_flag, p.err, kDevTimeoutProducer)) break;
        mbar_arrive_expect_tx(full_bar(s), STAGE_BYTES);
        const uint32_t a_dst = smem_base + s * STAGE_BYTES;
        const uint32_t b_dst = a_dst + A_TILE;
        if (kb < p.kb_main) {
          tma_load_2d(a_dst, tmx, kb * BK, m0, full_bar(s));
          tma_load_2d(b_dst, &tm_w, kb * BK, n0, full_bar(s));
        } else {
          const int kl = kb - p.kb_main;
          tma_load_2d(a_dst, &tm_u, kl * BK, m0, full_bar(s));
          tma_load_2d(b_dst, &tm_b, kl * BK, n0, full_bar(s));
        }
        ++issued;
      }
      // copies still in flight must land before the CTA's shared memory is released
      const int first = issued > STAGES ? issued - STAGES : 0;
      for (int kb = first; kb < issued; ++kb) {
        volatile int no_abort = 0;
        mbar_wait_bounded(full_bar(kb % STAGES), (kb / STAGES) & 1, &no_abort, p.err,
                          kDevTimeoutDrain);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------ MMA issuer
      bool ok = true;
      for (int kb = 0; kb < total_kb && ok; ++kb) {
        if (kb == p.kb_main && mid_drain) {
          tc_commit(acc_full);  // y_off = x W^T is complete in TMEM
          if (!mbar_wait_bounded(acc_empty, 0, abort_flag, p.err, kDevTimeoutMma)) {
            ok = false;
            break;
          }
          tc_fence_after();
        }
        const int s = kb % STAGES;
        const uint32_t ph = (kb / STAGES) & 1;
        if (!mbar_wait_bounded(full_bar(s), ph, abort_flag, p.err, kDevTimeoutMma)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a_base = smem_base + s * STAGE_BYTES;
        const uint32_t b_base = a_base + A_TILE;
        int nsub = BK / 16;
        if (kb >= p.kb_main) {
          const int rem = p.r - (kb - p.kb_main) * BK;
          nsub = min(BK / 16, (rem + 15) / 16);
        }
        for (int k = 0; k < nsub; ++k) {
          tc_mma_bf16(tmem_base, smem_desc_sw128(a_base + k * 32), smem_desc_sw128(b_base + k * 32),
                      IDESC, (kb > 0 || k > 0) ? 1u : 0u);
        }
        tc_commit(empty_bar(s));
      }
      if (ok) tc_commit(acc_full);
      // every issued MMA has finished before TMEM is released
      tc_commit(mma_done);
      volatile int no_abort = 0;
      mbar_wait_bounded(mma_done, 0, &no_abort, p.err, kDevTimeoutDrain);
    }
    __syncwarp();
  } else {
    // -------------------------------------------------------------- epilogue
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const int m = m0 + row;
    const uint32_t tmem_row = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
    uint32_t phase = 0;
    bool ok = true;
    if (mid_drain) {
      ok = mbar_wait_bounded(acc_full, 0, abort_flag, p.err, kDevTimeoutEpilogue);
      if (ok) {
        tc_fence_after();
        drain(tmem_row, m, p.M, n0, p, p.y_off, nullptr);
        tc_fence_before();
        mbar_arrive(acc_empty);
        phase = 1;
      }
    }
    if (ok && mbar_wait_bounded(acc_full, phase, abort_flag, p.err, kDevTimeoutEpilogue)) {
      tc_fence_after();
      drain(tmem_row, m, p.M, n0, p, fin0, fin1);
    }
    tc_fence_before();
  }

  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
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

// 2-D bf16 tensor map over a row-major [rows, cols] matrix, box [box_rows, 64] with
// 128-byte swizzle; out-of-bounds elements read as zero.
static bool make_map(CUtensorMap* map, const void* base, int64_t rows, int64_t cols,
                     int box_rows) {
  EncodeTiledFn enc = get_encode_fn();
  if (enc == nullptr) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(tcgemm::BK), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                   box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

int launch_dual_lora_gemm_tc(const GemmArgs& a, cudaStream_t stream) {
  using namespace tcgemm;
  static bool attr_set = false;
  if (!attr_set) {
    if (cudaFuncSetAttribute(dual_lora_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             SMEM_BYTES) != cudaSuccess)
      return -1;
    attr_set = true;
  }
  CUtensorMap m_xoff, m_xon, m_w, m_u, m_b;
  const bool lora = a.r > 0;
  if (!make_map(&m_xoff, a.x_off, a.M, a.K, BM)) return -2;
  if (!make_map(&m_xon, a.shared_x ? a.x_off : a.x_on, a.M, a.K, BM)) return -2;
  if (!make_map(&m_w, a.W, a.N, a.K, BN)) return -2;
  if (lora) {
    if (!make_map(&m_u, a.u, a.M, a.r, BM)) return -2;
    if (!make_map(&m_b, a.B, a.N, a.r, BN)) return -2;
  } else {
    m_u = m_xoff;
    m_b = m_w;
  }
  Params p;
  p.M = static_cast<int>(a.M);
  p.N = static_cast<int>(a.N);
  p.K = static_cast<int>(a.K);
  p.kb_main = static_cast<int>((a.K + BK - 1) / BK);
  p.kb_lora = lora ? static_cast<int>((a.r + BK - 1) / BK) : 0;
  p.r = static_cast<int>(a.r);
  p.shared_x = a.shared_x ? 1 : 0;
  p.m_tiles = static_cast<int>((a.M + BM - 1) / BM);
  p.n_tiles = static_cast<int>((a.N + BN - 1) / BN);
  p.y_off = a.y_off;
  p.y_on = a.y_on;
  p.out_f32 = a.out_f32;
  p.err = a.err;
  const int streams = a.shared_x ? 1 : 2;
  const unsigned grid = static_cast<unsigned>(p.m_tiles) * p.n_tiles * streams;
  dual_lora_gemm_kernel<<<grid, NUM_THREADS, SMEM_BYTES, stream>>>(m_xoff, m_xon, m_w, m_u, m_b, p);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace hydra
