// Skinny LoRA kernels:
//  * lora_down: u = s * (x_on A^T), bf16 [M, r]; the rank-r down-projection of the
//    LoRA update (§2 Stage 3: LoRA on all linear layers), with the scale folded in fp32
//    before the bf16 rounding. It is the operand of the LoRA-up MMA of the tcgen05
//    kernel and of the GEMV below. (Uses mma.sync: a skinny product far too narrow for a
//    128-row tcgen05 tile to stay busy.)
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
//
// u[M, r] = bf16(s * x A^T) as a skinny matrix product on the tensor cores (mma.sync
// m16n8k16, bf16 in, fp32 accumulate): one CTA per 16 token rows and per 64 ranks; its 8
// warps split K, load their fragments straight from global memory (each 32-byte row
// segment is read whole by four lanes) and reduce the 8 partial tiles in shared memory.

constexpr int kDownWarps = 8;

__device__ __forceinline__ uint32_t ld_pair(const __nv_bfloat16* p, bool ok) {
  return ok ? __ldg(reinterpret_cast<const uint32_t*>(p)) : 0u;
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
                     __nv_bfloat16* __restrict__ u) {
  __shared__ float red[kDownWarps][16][NT * 8 + 1];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int g = lane >> 2, c = lane & 3;
  const int row0 = blockIdx.x * 16;
  const int n_base = blockIdx.y * NT * 8;
  // this warp's K range, in whole k-steps of 16
  const int ksteps = (K + 15) / 16;
  const int per = (ksteps + kDownWarps - 1) / kDownWarps;
  const int ks0 = warp * per;
  const int ks1 = min(ksteps, ks0 + per);

  const bool r_lo = row0 + g < M, r_hi = row0 + g + 8 < M;
  const __nv_bfloat16* x_lo = x + static_cast<size_t>(r_lo ? row0 + g : 0) * K;
  const __nv_bfloat16* x_hi = x + static_cast<size_t>(r_hi ? row0 + g + 8 : 0) * K;
  const __nv_bfloat16* a_row[NT];
  bool a_ok[NT];
#pragma unroll
  for (int t = 0; t < NT; ++t) {
    const int n = n_base + t * 8 + g;
    a_ok[t] = n < r;
    a_row[t] = A + static_cast<size_t>(a_ok[t] ? n : 0) * K;
  }
  float d[NT][4];
#pragma unroll
  for (int t = 0; t < NT; ++t) d[t][0] = d[t][1] = d[t][2] = d[t][3] = 0.f;

#pragma unroll 4
  for (int ks = ks0; ks < ks1; ++ks) {
    const int k0 = ks * 16 + 2 * c;
    const int k1 = k0 + 8;
    const bool v0 = k0 < K, v1 = k1 < K;
    uint32_t a[4];
    a[0] = ld_pair(x_lo + k0, r_lo && v0);
    a[1] = ld_pair(x_hi + k0, r_hi && v0);
    a[2] = ld_pair(x_lo + k1, r_lo && v1);
    a[3] = ld_pair(x_hi + k1, r_hi && v1);
#pragma unroll
    for (int t = 0; t < NT; ++t) {
      const uint32_t b0 = ld_pair(a_row[t] + k0, a_ok[t] && v0);
      const uint32_t b1 = ld_pair(a_row[t] + k1, a_ok[t] && v1);
      mma_bf16_16816(d[t], a, b0, b1);
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
    const int m = row0 + rr, n = n_base + cc;
    if (m < M && n < r) u[static_cast<size_t>(m) * r + n] = __float2bfloat16_rn(s * v);
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
  const dim3 block(32 * kDownWarps);
  const auto* xp = static_cast<const __nv_bfloat16*>(x);
  const auto* ap = static_cast<const __nv_bfloat16*>(A);
  auto* up = static_cast<__nv_bfloat16*>(u);
  const unsigned gx = static_cast<unsigned>((M + 15) / 16);
  if (r <= 8) {
    lora_down_kernel<1><<<dim3(gx, 1), block, 0, stream>>>(xp, static_cast<int>(M), static_cast<int>(K), ap, static_cast<int>(r), s, up);
  } else if (r <= 16) {
    lora_down_kernel<2><<<dim3(gx, 1), block, 0, stream>>>(xp, static_cast<int>(M), static_cast<int>(K), ap, static_cast<int>(r), s, up);
  } else if (r <= 32) {
    lora_down_kernel<4><<<dim3(gx, 1), block, 0, stream>>>(xp, static_cast<int>(M), static_cast<int>(K), ap, static_cast<int>(r), s, up);
  } else {
    lora_down_kernel<8><<<dim3(gx, static_cast<unsigned>((r + 63) / 64)), block, 0, stream>>>(
        xp, static_cast<int>(M), static_cast<int>(K), ap, static_cast<int>(r), s, up);
  }
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
