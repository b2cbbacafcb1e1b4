// Certified decode for callers that cannot allocate device memory.
//
// ebd_certified_decode keeps its split-K partial records in a workspace the
// caller allocates.  Some callers have no way to do that: serving stacks that
// lay out every device buffer at start-up and forbid cudaMalloc afterwards
// (an allocation can synchronise the device and break a pre-planned memory
// pool), and plugin hosts that hand a custom operator its input and output
// buffers but no allocator.  ebd_certified_decode_static runs the very same
// decode with its scratch in a fixed-size array that belongs to the library
// itself, so the caller passes only inputs and outputs.
//
// The array is a file-scope __device__ variable: every GPU on which the
// library's device code is loaded holds these bytes until the process exits.
// Host code cannot use the array's name as a device address, so the address
// is looked up per device with cudaGetSymbolAddress (with that device
// current) the first time the entry point runs on it, and cached.
#include <cuda_runtime.h>

#include <mutex>

#include "decode.cuh"
#include "internal.h"

namespace ebd {

constexpr size_t kStaticScratchBytes = (size_t)16 << 20;  // 16 MiB per device
constexpr int kMaxStaticDevices = 64;

static __device__ __align__(256) unsigned char g_decode_scratch[kStaticScratchBytes];

static std::mutex g_scratch_mu;
static void* g_scratch_addr[kMaxStaticDevices] = {nullptr};

// Device address of g_decode_scratch on the current device (set up once per device).
static ebd_status static_scratch_address(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return EBD_ERR_CUDA;
  if (dev < 0 || dev >= kMaxStaticDevices) return EBD_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_decode_scratch);
    if (e != cudaSuccess || p == nullptr) return EBD_ERR_CUDA;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return EBD_OK;
}

}  // namespace ebd

using namespace ebd;

extern "C" ebd_status ebd_certified_decode_static(
    ebd_dtype dtype, int32_t batch, int32_t n_kv_heads, int32_t group, int32_t head_dim,
    const void* Q, const void* K_c, const void* V_c, const float* logw_c, const int32_t* n_kept,
    int32_t capacity, float delta, float eps0, ebd_range_mode range_mode, float* y, float* lse,
    float* var_hat, float* b_t, float* radius, int32_t* dev_status, void* stream) {
  // Same size query the workspace entry point uses; refuse before enqueueing.
  const size_t need =
      ebd_decode_workspace_bytes(dtype, batch, n_kv_heads, group, head_dim, capacity);
  if (need > kStaticScratchBytes) return EBD_ERR_CAPACITY;
  void* scratch = nullptr;
  const ebd_status st = static_scratch_address(&scratch);
  if (st != EBD_OK) return st;
  // Nothing in the scratch has to start at zero: the decode writes every
  // partial record before its reduce reads it, within the same call.
  return ebd_certified_decode(dtype, batch, n_kv_heads, group, head_dim, Q, K_c, V_c, logw_c,
                              n_kept, capacity, delta, eps0, range_mode, y, lse, var_hat, b_t,
                              radius, dev_status, scratch, kStaticScratchBytes, stream);
}
