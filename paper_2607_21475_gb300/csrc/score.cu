// E0: accumulated-attention importance scores (Appendix B of the paper,
// H2O-style accumulated attention from observation queries):
//     s_j = sum_r softmax_j(q_r . K^T / sqrt(d))
// over the R observation rows of a KV head's query group.
//
// Two passes per (batch row, KV head) unit:
//   pass 1  lse_r = log sum_j exp(q_r . k_j / sqrt(d))      (one warp per row)
//   pass 2  s_j   = sum_r exp(q_r . k_j / sqrt(d) - lse_r)   (one thread per key)
// Pass 2 owns each key column, so the sums are deterministic (no atomics).
#include <cuda_runtime.h>
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace ebd {

constexpr int kLseWarps = 8;
constexpr int kColThreads = 128;
constexpr int kColRows = 16;

template <typename T, int D>
__global__ void __launch_bounds__(kLseWarps * 32) score_lse_kernel(const T* __restrict__ q_obs,
                                                                   const T* __restrict__ K,
                                                                   int n_ctx, int n_obs,
                                                                   float* __restrict__ lse) {
  __shared__ float qs[kLseWarps][D];
  const int unit = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.y * kLseWarps + warp;
  const bool active = r < n_obs;
  const float scale = rsqrtf((float)D);
  if (active) {
    const T* q = q_obs + ((size_t)unit * n_obs + r) * D;
    for (int e = lane; e < D; e += 32) qs[warp][e] = to_f32(q[e]) * scale;
  }
  __syncwarp();
  if (!active) return;
  const T* Ku = K + (size_t)unit * n_ctx * D;
  float M = -INFINITY, S = 0.f;
  for (int j = lane; j < n_ctx; j += 32) {
    const T* kj = Ku + (size_t)j * D;
    float x = 0.f;
#pragma unroll 16
    for (int e = 0; e < D; ++e) x = fmaf(qs[warp][e], to_f32(kj[e]), x);
    if (x > M) {
      S = S * expf(M - x) + 1.f;
      M = x;
    } else {
      S += expf(x - M);
    }
  }
  // combine the lanes' (M, S)
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float Mo = __shfl_xor_sync(0xffffffffu, M, o);
    const float So = __shfl_xor_sync(0xffffffffu, S, o);
    const float Mn = fmaxf(M, Mo);
    S = (M == -INFINITY ? 0.f : S * expf(M - Mn)) + (Mo == -INFINITY ? 0.f : So * expf(Mo - Mn));
    M = Mn;
  }
  if (lane == 0) lse[(size_t)unit * n_obs + r] = M + logf(S);
}

template <typename T, int D>
__global__ void __launch_bounds__(kColThreads) score_col_kernel(const T* __restrict__ q_obs,
                                                                const T* __restrict__ K,
                                                                int n_ctx, int n_obs,
                                                                const float* __restrict__ lse,
                                                                float* __restrict__ scores) {
  extern __shared__ float smem[];
  float* ks = smem;                             // [kColThreads][D + 1]
  float* qs = smem + kColThreads * (D + 1);     // [kColRows][D]
  float* ls = qs + kColRows * D;                // [kColRows]
  const int unit = blockIdx.x;
  const int j0 = blockIdx.y * kColThreads;
  const int t = threadIdx.x;
  const float scale = rsqrtf((float)D);
  const T* Ku = K + (size_t)unit * n_ctx * D;
  for (int x = t; x < kColThreads * D; x += kColThreads) {
    const int row = x / D, e = x - row * D;
    const int j = j0 + row;
    ks[row * (D + 1) + e] = j < n_ctx ? to_f32(Ku[(size_t)j * D + e]) : 0.f;
  }
  float acc = 0.f;
  const T* Qu = q_obs + (size_t)unit * n_obs * D;
  for (int r0 = 0; r0 < n_obs; r0 += kColRows) {
    __syncthreads();
    for (int x = t; x < kColRows * D; x += kColThreads) {
      const int row = x / D, e = x - row * D;
      qs[x] = (r0 + row < n_obs) ? to_f32(Qu[(size_t)(r0 + row) * D + e]) * scale : 0.f;
    }
    for (int x = t; x < kColRows; x += kColThreads)
      ls[x] = (r0 + x < n_obs) ? lse[(size_t)unit * n_obs + r0 + x] : INFINITY;
    __syncthreads();
    const int nr = min(kColRows, n_obs - r0);
    for (int rr = 0; rr < nr; ++rr) {
      float x = 0.f;
#pragma unroll 16
      for (int e = 0; e < D; ++e) x = fmaf(qs[rr * D + e], ks[t * (D + 1) + e], x);
      acc += expf(x - ls[rr]);
    }
  }
  if (j0 + t < n_ctx) scores[(size_t)unit * n_ctx + j0 + t] = acc;
}

template <typename T, int D>
static ebd_status launch_score_t(int units, int n_ctx, int n_obs, const void* q_obs,
                                 const void* K, float* scores, float* lse, cudaStream_t s) {
  dim3 g1(units, (n_obs + kLseWarps - 1) / kLseWarps);
  score_lse_kernel<T, D><<<g1, kLseWarps * 32, 0, s>>>((const T*)q_obs, (const T*)K, n_ctx, n_obs,
                                                       lse);
  ebd_status st = launch_status();
  if (st != EBD_OK) return st;
  const size_t smem = (size_t)(kColThreads * (D + 1) + kColRows * D + kColRows) * sizeof(float);
  if (cudaFuncSetAttribute(score_col_kernel<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem) != cudaSuccess)
    return EBD_ERR_CUDA;
  dim3 g2(units, (n_ctx + kColThreads - 1) / kColThreads);
  score_col_kernel<T, D><<<g2, kColThreads, smem, s>>>((const T*)q_obs, (const T*)K, n_ctx, n_obs,
                                                       lse, scores);
  return launch_status();
}

ebd_status launch_score(ebd_dtype dtype, int batch, int n_kv_heads, int head_dim, int n_ctx,
                        int n_obs, const void* q_obs, const void* K, float* scores,
                        float* lse_ws, int32_t* dev_status, cudaStream_t s) {
  const int units = batch * n_kv_heads;
  if (units > 0x7fffffff || n_obs > 4096 || n_obs < 1) return EBD_ERR_UNSUPPORTED;
  if (score_tc_supported(dtype, head_dim, n_obs, q_obs, K))
    return launch_score_tc(units, head_dim, n_ctx, n_obs, q_obs, K, scores, lse_ws, dev_status, s);
  if (score_mma_supported(dtype, head_dim, q_obs, K) && units <= 65535 &&
      (n_ctx + 63) / 64 <= 65535)
    return launch_score_mma(units, head_dim, n_ctx, n_obs, q_obs, K, scores, lse_ws, dev_status, s);
  if ((n_obs + kLseWarps - 1) / kLseWarps > 65535 || (n_ctx + kColThreads - 1) / kColThreads > 65535)
    return EBD_ERR_UNSUPPORTED;
  if (dtype == EBD_BF16) {
    if (head_dim == 128) return launch_score_t<__nv_bfloat16, 128>(units, n_ctx, n_obs, q_obs, K, scores, lse_ws, s);
    if (head_dim == 64) return launch_score_t<__nv_bfloat16, 64>(units, n_ctx, n_obs, q_obs, K, scores, lse_ws, s);
  } else if (dtype == EBD_F32) {
    if (head_dim == 128) return launch_score_t<float, 128>(units, n_ctx, n_obs, q_obs, K, scores, lse_ws, s);
    if (head_dim == 64) return launch_score_t<float, 64>(units, n_ctx, n_obs, q_obs, K, scores, lse_ws, s);
  }
  return EBD_ERR_UNSUPPORTED;
}

}  // namespace ebd

using namespace ebd;

extern "C" size_t ebd_score_workspace_bytes(int32_t batch, int32_t n_kv_heads, int32_t n_obs) {
  if (batch < 1 || n_kv_heads < 1 || n_obs < 1) return 0;
  return align_up((size_t)batch * n_kv_heads * n_obs * sizeof(float), 256);
}

extern "C" ebd_status ebd_score(ebd_dtype dtype, int32_t batch, int32_t n_kv_heads,
                                int32_t head_dim, int32_t n_ctx, int32_t n_obs,
                                const void* q_obs, const void* K, float* scores, void* workspace,
                                size_t ws_bytes, void* stream) {
  if (batch < 1 || n_kv_heads < 1 || n_ctx < 1 || n_obs < 1 || !q_obs || !K || !scores)
    return EBD_ERR_INVALID;
  if (dtype != EBD_F32 && dtype != EBD_BF16) return EBD_ERR_INVALID;
  if (!workspace || ws_bytes < ebd_score_workspace_bytes(batch, n_kv_heads, n_obs))
    return EBD_ERR_CAPACITY;
  return launch_score(dtype, batch, n_kv_heads, head_dim, n_ctx, n_obs, q_obs, K, scores,
                      (float*)workspace, nullptr, (cudaStream_t)stream);
}
