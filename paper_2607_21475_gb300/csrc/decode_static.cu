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
// is looked up with cudaGetSymbolAddress (with the device current) the first
// time the entry point runs on a device, and cached together with the CUDA
// context that was current then; a call under another context (a
// driver-API context, or the new primary context after cudaDeviceReset)
// looks it up again.
#include <cuda.h>
#include <cudaTypedefs.h>
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
static CUcontext g_scratch_ctx[kMaxStaticDevices] = {nullptr};

// The CUDA context current on this thread (nullptr if it cannot be read).
static CUcontext current_context() {
  static PFN_cuCtxGetCurrent_v4000 get = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      p = nullptr;
    return reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
  }();
  CUcontext c = nullptr;
  if (get == nullptr || get(&c) != CUDA_SUCCESS) return nullptr;
  return c;
}

// Device address of g_decode_scratch on the current device, looked up once per
// (device, context).
static ebd_status static_scratch_address(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return EBD_ERR_CUDA;
  if (dev < 0 || dev >= kMaxStaticDevices) return EBD_ERR_UNSUPPORTED;
  // (with no context current yet ctx is null and the address is looked up
  // again, cudaGetSymbolAddress making the primary context current)
  const CUcontext ctx = current_context();
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_addr[dev] == nullptr || ctx == nullptr || ctx != g_scratch_ctx[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_decode_scratch);
    if (e != cudaSuccess || p == nullptr) return EBD_ERR_CUDA;
    g_scratch_addr[dev] = p;
    g_scratch_ctx[dev] = ctx;
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
  // The workspace entry point's argument checks first (same status for the
  // same bad request), then its size query; refuse before enqueueing.
  const ebd_status arg = check_decode_args(dtype, batch, n_kv_heads, group, head_dim, Q, K_c,
                                           V_c, logw_c, n_kept, capacity, delta, eps0,
                                           range_mode, y, lse, var_hat, b_t, radius);
  if (arg != EBD_OK) return arg;
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
