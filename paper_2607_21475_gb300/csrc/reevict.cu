// The decode-time life of a compact cache: tokens generated after an
// eviction join it with pi = 1, and every T_r decode steps the resident cache
// is evicted again with fresh tail draws (the redraw-every-T_r-steps schedule
// of the paper's anytime argument, Section 4 and its appendix).  A token kept
// by both designs has inclusion probability pi_1 pi_2 (independent Poisson
// designs compose), so its log(1/pi) is the sum of the two rounds' values, and
// it keeps its original token position.
#include <cuda_runtime.h>

#include "common.cuh"
#include "internal.h"

namespace ebd {

constexpr int kAppendWarps = 8;
constexpr int kComposeThreads = 256;

// One warp per unit: row n_kept of K_c/V_c <- the new key/value (16-byte
// chunks), log(1/pi) = 0, token position; n_kept + 1.
__global__ void __launch_bounds__(kAppendWarps * 32)
    append_kernel(const uint4* __restrict__ k_new, const uint4* __restrict__ v_new,
                  const int32_t* __restrict__ positions, int units, int n_kv_heads, int cpr,
                  int cap, uint4* __restrict__ K_c, uint4* __restrict__ V_c,
                  float* __restrict__ logw_c, int32_t* __restrict__ idx_c,
                  int32_t* __restrict__ n_kept, int32_t* dev_status) {
  // a decode launched next as a programmatic dependent may start its launch
  // now; it waits for this kernel's writes before reading the cache
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int unit = blockIdx.x * kAppendWarps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (unit >= units) return;
  const int n = max(n_kept[unit], 0);
  __syncwarp();
  if (n < cap) {
    const size_t dst = ((size_t)unit * cap + n) * cpr;
    for (int c = lane; c < 2 * cpr; c += 32) {
      if (c < cpr) K_c[dst + c] = k_new[(size_t)unit * cpr + c];
      else V_c[dst + c - cpr] = v_new[(size_t)unit * cpr + c - cpr];
    }
    if (lane == 0) {
      logw_c[(size_t)unit * cap + n] = 0.f;
      idx_c[(size_t)unit * cap + n] = positions[unit / n_kv_heads];
    }
  } else if (lane == 0) {
    raise_status(dev_status, EBD_DEV_CAPACITY);
  }
  if (lane == 0) n_kept[unit] = n + 1;
}

// After the re-eviction's select (resident positions and this round's
// log(1/pi) in idx_out/logw_out) and row gather: compose with the first round.
__global__ void __launch_bounds__(kComposeThreads)
    compose_kernel(const float* __restrict__ logw_in, const int32_t* __restrict__ idx_in,
                   int cap_in, const int32_t* __restrict__ n_kept_out, int cap_out,
                   float* __restrict__ logw_out, int32_t* __restrict__ idx_out) {
  const int unit = blockIdx.y;
  const int n = min(max(n_kept_out[unit], 0), cap_out);
  for (int p = blockIdx.x * kComposeThreads + threadIdx.x; p < n;
       p += gridDim.x * kComposeThreads) {
    const size_t o = (size_t)unit * cap_out + p;
    const int j = idx_out[o];  // resident position in the input cache, < cap_in
    const size_t i = (size_t)unit * cap_in + j;
    logw_out[o] += logw_in[i];
    idx_out[o] = idx_in[i];
  }
}

}  // namespace ebd

using namespace ebd;

extern "C" ebd_status ebd_append(ebd_dtype dtype, int32_t batch, int32_t n_kv_heads,
                                 int32_t head_dim, const void* k_new, const void* v_new,
                                 const int32_t* positions, void* K_c, void* V_c, float* logw_c,
                                 int32_t* idx_c, int32_t* n_kept, int32_t capacity,
                                 int32_t* dev_status, void* stream) {
  if (dtype != EBD_F32 && dtype != EBD_BF16) return EBD_ERR_INVALID;
  if (batch < 1 || n_kv_heads < 1 || head_dim < 1 || capacity < 1) return EBD_ERR_INVALID;
  if (!k_new || !v_new || !positions || !K_c || !V_c || !logw_c || !idx_c || !n_kept ||
      !dev_status)
    return EBD_ERR_INVALID;
  const int eb = dtype == EBD_F32 ? 4 : 2;
  if ((head_dim * eb) % 16 != 0) return EBD_ERR_UNSUPPORTED;
  if (!aligned16(k_new) || !aligned16(v_new) || !aligned16(K_c) || !aligned16(V_c))
    return EBD_ERR_INVALID;
  const long long units = (long long)batch * n_kv_heads;
  if (units > 0x7fffffffLL) return EBD_ERR_UNSUPPORTED;
  const int cpr = head_dim * eb / 16;
  const int blocks = (int)((units + kAppendWarps - 1) / kAppendWarps);
  append_kernel<<<blocks, kAppendWarps * 32, 0, (cudaStream_t)stream>>>(
      (const uint4*)k_new, (const uint4*)v_new, positions, (int)units, n_kv_heads, cpr, capacity,
      (uint4*)K_c, (uint4*)V_c, logw_c, idx_c, n_kept, dev_status);
  return launch_status();
}

extern "C" ebd_status ebd_reevict(const ebd_design* design, ebd_dtype dtype, const float* scores,
                                  const void* K_in, const void* V_in, const float* logw_in,
                                  const int32_t* idx_in, const int32_t* n_kept_in,
                                  int32_t cap_in, void* K_out, void* V_out, float* logw_out,
                                  int32_t* idx_out, int32_t* n_kept_out, int32_t cap_out,
                                  int32_t* dev_status, void* stream) {
  ebd_status st = check_design(design);
  if (st != EBD_OK) return st;
  if (dtype != EBD_F32 && dtype != EBD_BF16) return EBD_ERR_INVALID;
  if (cap_in < 1 || cap_out < 1 || design->n_ctx != cap_in) return EBD_ERR_INVALID;
  if (!scores || !K_in || !V_in || !logw_in || !idx_in || !n_kept_in || !K_out || !V_out ||
      !logw_out || !idx_out || !n_kept_out || !dev_status)
    return EBD_ERR_INVALID;
  if (K_out == K_in || V_out == V_in || logw_out == logw_in || idx_out == idx_in ||
      n_kept_out == n_kept_in)
    return EBD_ERR_INVALID;
  const int eb = dtype == EBD_F32 ? 4 : 2;
  if (design->head_dim < 1 || (design->head_dim * eb) % 16 != 0) return EBD_ERR_UNSUPPORTED;
  if (!aligned16(K_in) || !aligned16(V_in) || !aligned16(K_out) || !aligned16(V_out))
    return EBD_ERR_INVALID;
  const int units = design->batch * design->n_kv_heads;
  if (units > 65535) return EBD_ERR_UNSUPPORTED;
  cudaStream_t s = (cudaStream_t)stream;
  // this round's design over each unit's resident rows (positions 0 .. n_kept_in - 1)
  st = launch_select(design, scores, n_kept_in, nullptr, nullptr, idx_out, logw_out, n_kept_out,
                     cap_out, dev_status, s);
  if (st != EBD_OK) return st;
  st = launch_gather(design, dtype, K_in, V_in, idx_out, n_kept_out, cap_out, K_out, V_out, s);
  if (st != EBD_OK) return st;
  int bx = (cap_out + kComposeThreads - 1) / kComposeThreads;
  if (bx > 65535) bx = 65535;
  compose_kernel<<<dim3(bx, units), kComposeThreads, 0, s>>>(logw_in, idx_in, cap_in, n_kept_out,
                                                             cap_out, logw_out, idx_out);
  return launch_status();
}
