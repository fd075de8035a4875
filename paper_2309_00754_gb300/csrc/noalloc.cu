// hydra_lora_linear_noalloc: the dual-output LoRA linear for callers that cannot allocate
// device memory themselves, e.g. a plugin inside a host framework that owns the device
// memory pool and hands it only input and output buffers, or a latency-critical caller
// that cannot afford cudaMalloc/cudaFree, which may synchronise the device.
//
// hydra_lora_linear keeps u = s x_on A^T in a caller-provided workspace. This variant
// keeps u instead in the file-scope device array below (4 MiB), which every device that
// loads the library holds until the process exits. Nothing here calls cudaMalloc,
// cudaFree or any allocating library routine.
//
// Device set-up: the first call on a device, with that device current, resolves the
// array's device address with cudaGetSymbolAddress and caches it. Make that first call
// before any stream capture on the device.
//
// All calls share the one array and it keeps the last call's contents. Every element of u
// that a call reads is written earlier in the same call, so nothing has to start at zero.
// Calls whose work overlaps on the GPU (on different streams, or from different host
// threads without ordering) race on the array.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "../../include/hydra.h"

namespace {

static __device__ __align__(256) uint16_t g_noalloc_u[HYDRA_NOALLOC_MAX_U_ELEMS];

constexpr int kMaxDevices = 64;
void* g_u_ptr[kMaxDevices] = {nullptr};
std::mutex g_setup_mutex;

// Device address of g_noalloc_u on the current device (set up once per device).
void* scratch_ptr() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (g_u_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_u) != cudaSuccess) return nullptr;
    g_u_ptr[dev] = p;
  }
  return g_u_ptr[dev];
}

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" hydra_status hydra_lora_linear_noalloc(const void* x_off, const void* x_on, int64_t M,
                                                  int64_t K, int64_t N, const void* W,
                                                  const void* A, const void* B, int64_t r,
                                                  float s, void* y_off, void* y_on,
                                                  int out_dtype, void* stream) {
  // the same argument rules as hydra_lora_linear, all checked before anything is launched
  if (x_off == nullptr || W == nullptr) return HYDRA_ERR_NULL;
  if (y_off == nullptr && y_on == nullptr) return HYDRA_ERR_NULL;
  if (out_dtype != HYDRA_BF16 && out_dtype != HYDRA_F32) return HYDRA_ERR_RANGE;
  if (M < 0 || K < 8 || N < 8 || M >= (1LL << 31) || K >= (1LL << 31) || N >= (1LL << 31))
    return HYDRA_ERR_SHAPE;
  if (K % 8 != 0 || N % 8 != 0) return HYDRA_ERR_ALIGN;
  if (r < 0 || r > 256) return HYDRA_ERR_SHAPE;
  if (r > 0 && r % 8 != 0) return HYDRA_ERR_ALIGN;
  const bool shared_x = (x_on == nullptr || x_on == x_off);
  if (!aligned16(x_off) || (!shared_x && !aligned16(x_on)) || !aligned16(W) ||
      !aligned16(y_off) || !aligned16(y_on))
    return HYDRA_ERR_ALIGN;
  const bool lora = r > 0 && y_on != nullptr;
  if (lora) {
    if (A == nullptr || B == nullptr) return HYDRA_ERR_NULL;
    if (!aligned16(A) || !aligned16(B)) return HYDRA_ERR_ALIGN;
    // u must fit the static array
    if (M * r > static_cast<int64_t>(HYDRA_NOALLOC_MAX_U_ELEMS)) return HYDRA_ERR_SHAPE;
  }
  if (M == 0) return HYDRA_OK;
  if (!lora)
    return hydra_dual_linear(x_off, x_on, M, K, N, W, nullptr, nullptr, 0, y_off, y_on, out_dtype,
                             0, stream);
  void* u = scratch_ptr();
  if (u == nullptr) return HYDRA_ERR_CUDA;
  const hydra_status st = hydra_lora_down(shared_x ? x_off : x_on, M, K, A, r, s, u, stream);
  if (st != HYDRA_OK) return st;
  return hydra_dual_linear(x_off, x_on, M, K, N, W, u, B, r, y_off, y_on, out_dtype, 0, stream);
}
