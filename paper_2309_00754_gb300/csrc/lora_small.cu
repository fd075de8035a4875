// Skinny LoRA kernels on the CUDA cores:
//  * lora_down: u = s * (x_on A^T), bf16 [M, r]; the rank-r down-projection of the
//    LoRA update (§2 Stage 3: LoRA on all linear layers), with the scale folded in fp32
//    before the bf16 rounding. It is the operand of the LoRA-up MMA of the tensor-core
//    kernel and of the GEMV below.
//  * dual_lora_gemv: the dual-output linear for decode-shaped inputs (at most 16 token
//    rows over both streams), y_off = x_off W^T, y_on = x_on W^T + u B^T. One warp owns two
//    rows of W and streams them once with 128-bit loads; the token rows are re-read from
//    L1. Used where a 128-row tensor-core tile would be almost empty.
#include "common.cuh"
#include "kernels.h"

namespace hydra {
namespace {

__device__ __forceinline__ void unpack8(const uint4& v, float (&f)[8]) {
  float2 a = unpack_bf16x2(v.x), b = unpack_bf16x2(v.y), c = unpack_bf16x2(v.z),
         d = unpack_bf16x2(v.w);
  f[0] = a.x; f[1] = a.y; f[2] = b.x; f[3] = b.y;
  f[4] = c.x; f[5] = c.y; f[6] = d.x; f[7] = d.y;
}

__device__ __forceinline__ float dot8(const float (&a)[8], const float (&b)[8]) {
  float s = a[0] * b[0];
#pragma unroll
  for (int i = 1; i < 8; ++i) s = fmaf(a[i], b[i], s);
  return s;
}

// ---------------------------------------------------------------- lora_down

constexpr int kDownRows = 4;   // token rows per warp
constexpr int kDownRJ = 16;    // LoRA ranks per CTA column (grid.y covers r)

__global__ void __launch_bounds__(256)
    lora_down_kernel(const __nv_bfloat16* __restrict__ x, int M, int K,
                     const __nv_bfloat16* __restrict__ A, int r, float s,
                     __nv_bfloat16* __restrict__ u) {
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int row0 = (blockIdx.x * 8 + warp) * kDownRows;
  const int j0 = blockIdx.y * kDownRJ;
  if (row0 >= M) return;
  float acc[kDownRows][kDownRJ];
#pragma unroll
  for (int i = 0; i < kDownRows; ++i)
#pragma unroll
    for (int j = 0; j < kDownRJ; ++j) acc[i][j] = 0.f;

  for (int k = lane * 8; k < K; k += 256) {
    float xv[kDownRows][8];
#pragma unroll
    for (int i = 0; i < kDownRows; ++i) {
      if (row0 + i < M) {
        unpack8(__ldg(reinterpret_cast<const uint4*>(x + static_cast<size_t>(row0 + i) * K + k)),
                xv[i]);
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) xv[i][e] = 0.f;
      }
    }
#pragma unroll
    for (int j = 0; j < kDownRJ; ++j) {
      if (j0 + j < r) {
        float av[8];
        unpack8(__ldg(reinterpret_cast<const uint4*>(A + static_cast<size_t>(j0 + j) * K + k)), av);
#pragma unroll
        for (int i = 0; i < kDownRows; ++i) acc[i][j] += dot8(xv[i], av);
      }
    }
  }
#pragma unroll
  for (int i = 0; i < kDownRows; ++i)
#pragma unroll
    for (int j = 0; j < kDownRJ; ++j) {
      float v = acc[i][j];
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
      acc[i][j] = v;
    }
#pragma unroll
  for (int i = 0; i < kDownRows; ++i)
#pragma unroll
    for (int j = 0; j < kDownRJ; ++j) {
      if (((i * kDownRJ + j) & 31) == lane && row0 + i < M && j0 + j < r)
        u[static_cast<size_t>(row0 + i) * r + j0 + j] = __float2bfloat16_rn(s * acc[i][j]);
    }
}

// ---------------------------------------------------------------- dual_lora_gemv

constexpr int kGemvNR = 2;  // W rows per warp

template <int MT>
__global__ void __launch_bounds__(256)
    dual_lora_gemv_kernel(const __nv_bfloat16* __restrict__ x_off,
                          const __nv_bfloat16* __restrict__ x_on, int M, int K, int N,
                          const __nv_bfloat16* __restrict__ W, const __nv_bfloat16* __restrict__ u,
                          const __nv_bfloat16* __restrict__ B, int r, void* y_off, void* y_on,
                          int out_f32, int shared_x) {
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int n0 = (blockIdx.x * 8 + warp) * kGemvNR;
  if (n0 >= N) return;
  // token rows: [0, M) from x_off; in the stacked case rows [M, 2M) from x_on
  const int rows = shared_x ? M : 2 * M;
  float acc[MT][kGemvNR];
#pragma unroll
  for (int i = 0; i < MT; ++i)
#pragma unroll
    for (int q = 0; q < kGemvNR; ++q) acc[i][q] = 0.f;

  for (int k = lane * 8; k < K; k += 256) {
    float wv[kGemvNR][8];
#pragma unroll
    for (int q = 0; q < kGemvNR; ++q) {
      if (n0 + q < N) {
        unpack8(__ldcs(reinterpret_cast<const uint4*>(W + static_cast<size_t>(n0 + q) * K + k)),
                wv[q]);
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) wv[q][e] = 0.f;
      }
    }
#pragma unroll
    for (int i = 0; i < MT; ++i) {
      if (i < rows) {
        const __nv_bfloat16* xr =
            (i < M) ? x_off + static_cast<size_t>(i) * K : x_on + static_cast<size_t>(i - M) * K;
        float xv[8];
        unpack8(__ldg(reinterpret_cast<const uint4*>(xr + k)), xv);
#pragma unroll
        for (int q = 0; q < kGemvNR; ++q) acc[i][q] += dot8(xv, wv[q]);
      }
    }
  }
#pragma unroll
  for (int i = 0; i < MT; ++i)
#pragma unroll
    for (int q = 0; q < kGemvNR; ++q) {
      float v = acc[i][q];
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
      acc[i][q] = v;
    }

  // LoRA-up on the on-stream rows: lanes split the rank dimension
  float lora[MT][kGemvNR];
#pragma unroll
  for (int i = 0; i < MT; ++i)
#pragma unroll
    for (int q = 0; q < kGemvNR; ++q) lora[i][q] = 0.f;
  if (u != nullptr) {
#pragma unroll
    for (int i = 0; i < MT; ++i) {
      if (i < M) {
#pragma unroll
        for (int q = 0; q < kGemvNR; ++q) {
          float v = 0.f;
          if (n0 + q < N) {
            for (int j = lane; j < r; j += 32)
              v = fmaf(__bfloat162float(u[static_cast<size_t>(i) * r + j]),
                       __bfloat162float(B[static_cast<size_t>(n0 + q) * r + j]), v);
          }
#pragma unroll
          for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
          lora[i][q] = v;
        }
      }
    }
  }

#pragma unroll
  for (int i = 0; i < MT; ++i)
#pragma unroll
    for (int q = 0; q < kGemvNR; ++q) {
      if (((i * kGemvNR + q) & 31) != lane || i >= rows || n0 + q >= N) continue;
      const int n = n0 + q;
      // (output, token row, value) for this accumulator
      void* dst0 = nullptr;
      void* dst1 = nullptr;
      int m;
      float v0, v1 = 0.f;
      if (shared_x) {
        m = i;
        dst0 = y_off;
        v0 = acc[i][q];
        dst1 = y_on;
        v1 = acc[i][q] + lora[i][q];
      } else if (i < M) {
        m = i;
        dst0 = y_off;
        v0 = acc[i][q];
      } else {
        m = i - M;
        dst0 = y_on;
        v0 = acc[i][q] + lora[m][q];
      }
      const size_t o = static_cast<size_t>(m) * N + n;
      if (out_f32) {
        if (dst0) reinterpret_cast<float*>(dst0)[o] = v0;
        if (dst1) reinterpret_cast<float*>(dst1)[o] = v1;
      } else {
        if (dst0) reinterpret_cast<__nv_bfloat16*>(dst0)[o] = __float2bfloat16_rn(v0);
        if (dst1) reinterpret_cast<__nv_bfloat16*>(dst1)[o] = __float2bfloat16_rn(v1);
      }
    }
}

template <int MT>
void launch_gemv_t(const GemmArgs& a, cudaStream_t stream) {
  const unsigned grid = static_cast<unsigned>((a.N + 8 * kGemvNR - 1) / (8 * kGemvNR));
  dual_lora_gemv_kernel<MT><<<grid, 256, 0, stream>>>(
      static_cast<const __nv_bfloat16*>(a.x_off),
      static_cast<const __nv_bfloat16*>(a.shared_x ? a.x_off : a.x_on), static_cast<int>(a.M),
      static_cast<int>(a.K), static_cast<int>(a.N), static_cast<const __nv_bfloat16*>(a.W),
      static_cast<const __nv_bfloat16*>(a.u), static_cast<const __nv_bfloat16*>(a.B),
      static_cast<int>(a.r), a.y_off, a.y_on, a.out_f32, a.shared_x ? 1 : 0);
}

}  // namespace

int launch_lora_down(const void* x, int64_t M, int64_t K, const void* A, int64_t r, float s,
                     void* u, cudaStream_t stream) {
  if (M == 0 || r == 0) return 0;
  dim3 grid(static_cast<unsigned>((M + 8 * kDownRows - 1) / (8 * kDownRows)),
            static_cast<unsigned>((r + kDownRJ - 1) / kDownRJ));
  lora_down_kernel<<<grid, 256, 0, stream>>>(
      static_cast<const __nv_bfloat16*>(x), static_cast<int>(M), static_cast<int>(K),
      static_cast<const __nv_bfloat16*>(A), static_cast<int>(r), s,
      static_cast<__nv_bfloat16*>(u));
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

int launch_dual_lora_gemv(const GemmArgs& a, cudaStream_t stream) {
  const int64_t rows = a.shared_x ? a.M : 2 * a.M;
  if (rows <= 1)
    launch_gemv_t<1>(a, stream);
  else if (rows <= 2)
    launch_gemv_t<2>(a, stream);
  else if (rows <= 4)
    launch_gemv_t<4>(a, stream);
  else if (rows <= 8)
    launch_gemv_t<8>(a, stream);
  else
    launch_gemv_t<16>(a, stream);
  return cudaPeekAtLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace hydra
