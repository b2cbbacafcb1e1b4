// Score queries and per-token variance contributions.
//
// Observation queries.  The paper's harness scores the cache from three query
// sets (Appendix, experimental details): strided prefill queries (H2O-style
// accumulated attention), the last 64 prefill positions (SnapKV-style
// observation window) or the question's positions (question-aware).  All three
// are rows of the prefill queries at chosen positions; ebd_gather_queries
// lays them out as the observation rows E0 consumes.
//
// Variance contributions.  Theorem 2's estimator is a sum over the retained
// tail, V_hat = sum_i (1 - pi_i) p_i^2 ||v_i - y_hat||^2 with p_i = w_i / N_hat;
// each term is one retained token's contribution.  The fine-grained probe of
// Section 5 ranks evicted 64-token blocks by the contribution of their retained
// neighbours; ebd_block_scores sums the contributions over blocks of original
// token positions.  A second pass over the compact cache (y_hat and log N_hat
// come from the certified decode), one warp per token of a split.
#include <cuda_runtime.h>

#include "common.cuh"
#include "internal.h"

namespace ebd {

constexpr int kCtbThreads = 128;
constexpr int kCtbWarps = kCtbThreads / 32;
constexpr int kCtbMaxG = 8;

// One warp per output row: q_obs[b, kvh, g * P + p] = Q[b, kvh * G + g, pos[p]].
__global__ void gather_queries_kernel(const uint4* __restrict__ Q, const int32_t* __restrict__ pos,
                                      int n_kv_heads, int group, int n_rows_q, int n_pos, int cpr,
                                      long long out_rows, uint4* __restrict__ q_obs) {
  const long long row = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= out_rows) return;
  const int P = n_pos;
  const long long unit = row / ((long long)group * P);
  const int rem = (int)(row - unit * group * P);
  const int g = rem / P, p = rem - g * P;
  const int b = (int)(unit / n_kv_heads), kvh = (int)(unit - (long long)b * n_kv_heads);
  const long long hq = (long long)b * n_kv_heads * group + (long long)kvh * group + g;
  const uint4* src = Q + ((size_t)hq * n_rows_q + pos[p]) * cpr;
  uint4* dst = q_obs + (size_t)row * cpr;
  for (int c = lane; c < cpr; c += 32) dst[c] = src[c];
}

// contrib[b, kvh * G + g, i] = (1 - pi_i) p_i^2 ||v_i - y_hat_g||^2 for the
// retained rows i < min(n_kept, cap) (0 for certain rows and rows past n_kept).
template <typename T, int D>
__global__ void __launch_bounds__(kCtbThreads)
    variance_contrib_kernel(const T* __restrict__ Qh, const T* __restrict__ Kc,
                            const T* __restrict__ Vc, const float* __restrict__ logw,
                            const int32_t* __restrict__ n_kept, const float* __restrict__ y,
                            const float* __restrict__ lse, int group, int cap,
                            int tokens_per_split, float* __restrict__ contrib) {
  constexpr int E = D / 32;
  const int unit = blockIdx.y, split = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = group;
  const int n = min(max(n_kept[unit], 0), cap);
  const int t0 = split * tokens_per_split;
  const int t1 = min(cap, t0 + tokens_per_split);
  const float scale = rsqrtf((float)D);
  const size_t hq0 = (size_t)unit * G;
  float q[kCtbMaxG][E], yv[kCtbMaxG][E], ls[kCtbMaxG];
#pragma unroll
  for (int g = 0; g < kCtbMaxG; ++g) {
#pragma unroll
    for (int j = 0; j < E; ++j) {
      q[g][j] = g < G ? to_f32(Qh[(hq0 + g) * D + lane + 32 * j]) * scale : 0.f;
      yv[g][j] = g < G ? y[(hq0 + g) * D + lane + 32 * j] : 0.f;
    }
    ls[g] = g < G ? lse[hq0 + g] : 0.f;
  }
  for (int t = t0 + warp; t < t1; t += kCtbWarps) {
    const float lwt = t < n ? logw[(size_t)unit * cap + t] : 0.f;
    if (!(lwt > 0.f)) {  // certain (pi = 1) or past n_kept: no contribution
      if (lane < G) contrib[(hq0 + lane) * cap + t] = 0.f;
      continue;
    }
    float k[E], v[E];
#pragma unroll
    for (int j = 0; j < E; ++j) {
      k[j] = to_f32(Kc[((size_t)unit * cap + t) * D + lane + 32 * j]);
      v[j] = to_f32(Vc[((size_t)unit * cap + t) * D + lane + 32 * j]);
    }
    const float omp = -expm1f(-lwt);  // 1 - pi
    float out = 0.f;
#pragma unroll
    for (int g = 0; g < kCtbMaxG; ++g) {
      if (g >= G) break;
      float dot = 0.f, dist = 0.f;
#pragma unroll
      for (int j = 0; j < E; ++j) {
        dot = fmaf(q[g][j], k[j], dot);
        const float dv = v[j] - yv[g][j];
        dist = fmaf(dv, dv, dist);
      }
      const float x = warp_sum(dot) + lwt;
      dist = warp_sum(dist);
      const float p = expf(x - ls[g]);  // w_i / N_hat
      if (lane == g) out = omp * p * p * dist;
    }
    if (lane < G) contrib[(hq0 + lane) * cap + t] = out;
  }
}

// out[b, kvh, k] = sum over the unit's G heads and retained rows whose
// original position lies in [k * block, (k + 1) * block).  idx_c is
// increasing, so each block's rows are one run, found by binary search and
// added in order (deterministic).
__global__ void block_scores_kernel(const float* __restrict__ contrib,
                                    const int32_t* __restrict__ idx_c,
                                    const int32_t* __restrict__ n_kept, int group, int cap,
                                    int block, int n_blocks, float* __restrict__ out) {
  const int unit = blockIdx.y;
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= n_blocks) return;
  const int n = min(max(n_kept[unit], 0), cap);
  const int32_t* ix = idx_c + (size_t)unit * cap;
  auto lower = [&](long long key) {
    int lo = 0, hi = n;
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if ((long long)ix[mid] < key) lo = mid + 1;
      else hi = mid;
    }
    return lo;
  };
  const int a0 = lower((long long)k * block), a1 = lower((long long)(k + 1) * block);
  float s = 0.f;
  for (int g = 0; g < group; ++g) {
    const float* c = contrib + ((size_t)unit * group + g) * cap;
    for (int i = a0; i < a1; ++i) s += c[i];
  }
  out[(size_t)unit * n_blocks + k] = s;
}

template <typename T, int D>
static ebd_status launch_contrib_t(int units, int group, int cap, const void* Q, const void* K_c,
                                   const void* V_c, const float* logw_c, const int32_t* n_kept,
                                   const float* y, const float* lse, float* contrib,
                                   cudaStream_t s) {
  const long long target = (long long)sm_count() * 8;
  long long splits = (target + units - 1) / units;
  const long long max_splits = (cap + 31) / 32;
  if (splits > max_splits) splits = max_splits;
  if (splits < 1) splits = 1;
  if (splits > 65535) splits = 65535;
  const int tps = (int)((cap + splits - 1) / splits);
  variance_contrib_kernel<T, D><<<dim3((unsigned)splits, units), kCtbThreads, 0, s>>>(
      (const T*)Q, (const T*)K_c, (const T*)V_c, logw_c, n_kept, y, lse, group, cap, tps, contrib);
  return launch_status();
}

}  // namespace ebd

using namespace ebd;

extern "C" ebd_status ebd_gather_queries(ebd_dtype dtype, int32_t batch, int32_t n_kv_heads,
                                         int32_t group, int32_t head_dim, int32_t n_rows_q,
                                         const void* Q, const int32_t* positions, int32_t n_pos,
                                         void* q_obs, void* stream) {
  if (dtype != EBD_F32 && dtype != EBD_BF16) return EBD_ERR_INVALID;
  if (batch < 1 || n_kv_heads < 1 || group < 1 || head_dim < 1 || n_rows_q < 1 || n_pos < 1 ||
      !Q || !positions || !q_obs)
    return EBD_ERR_INVALID;
  const int eb = dtype == EBD_F32 ? 4 : 2;
  if ((head_dim * eb) % 16 != 0) return EBD_ERR_UNSUPPORTED;
  if (!aligned16(Q) || !aligned16(q_obs)) return EBD_ERR_INVALID;
  const long long rows = (long long)batch * n_kv_heads * group * n_pos;
  const int per_block = 8;
  const long long blocks = (rows + per_block - 1) / per_block;
  if (blocks > 0x7fffffffLL) return EBD_ERR_UNSUPPORTED;
  gather_queries_kernel<<<(unsigned)blocks, per_block * 32, 0, (cudaStream_t)stream>>>(
      (const uint4*)Q, positions, n_kv_heads, group, n_rows_q, n_pos, head_dim * eb / 16, rows,
      (uint4*)q_obs);
  return launch_status();
}

extern "C" ebd_status ebd_variance_contributions(ebd_dtype dtype, int32_t batch,
                                                 int32_t n_kv_heads, int32_t group,
                                                 int32_t head_dim, const void* Q, const void* K_c,
                                                 const void* V_c, const float* logw_c,
                                                 const int32_t* n_kept, int32_t capacity,
                                                 const float* y, const float* lse, float* contrib,
                                                 void* stream) {
  if (dtype != EBD_F32 && dtype != EBD_BF16) return EBD_ERR_INVALID;
  if (batch < 1 || n_kv_heads < 1 || group < 1 || capacity < 1) return EBD_ERR_INVALID;
  if (!Q || !K_c || !V_c || !logw_c || !n_kept || !y || !lse || !contrib) return EBD_ERR_INVALID;
  if (group > kCtbMaxG || (head_dim != 64 && head_dim != 128)) return EBD_ERR_UNSUPPORTED;
  const long long units = (long long)batch * n_kv_heads;
  if (units > 65535) return EBD_ERR_UNSUPPORTED;
  cudaStream_t s = (cudaStream_t)stream;
  const int u = (int)units;
  if (dtype == EBD_F32) {
    if (head_dim == 64)
      return launch_contrib_t<float, 64>(u, group, capacity, Q, K_c, V_c, logw_c, n_kept, y, lse,
                                         contrib, s);
    return launch_contrib_t<float, 128>(u, group, capacity, Q, K_c, V_c, logw_c, n_kept, y, lse,
                                        contrib, s);
  }
  if (head_dim == 64)
    return launch_contrib_t<__nv_bfloat16, 64>(u, group, capacity, Q, K_c, V_c, logw_c, n_kept, y,
                                               lse, contrib, s);
  return launch_contrib_t<__nv_bfloat16, 128>(u, group, capacity, Q, K_c, V_c, logw_c, n_kept, y,
                                              lse, contrib, s);
}

extern "C" ebd_status ebd_block_scores(int32_t batch, int32_t n_kv_heads, int32_t group,
                                       const float* contrib, const int32_t* idx_c,
                                       const int32_t* n_kept, int32_t capacity, int32_t block,
                                       int32_t n_blocks, float* out, void* stream) {
  if (batch < 1 || n_kv_heads < 1 || group < 1 || capacity < 1 || block < 1 || n_blocks < 1 ||
      !contrib || !idx_c || !n_kept || !out)
    return EBD_ERR_INVALID;
  const long long units = (long long)batch * n_kv_heads;
  if (units > 65535) return EBD_ERR_UNSUPPORTED;
  const int threads = 128;
  block_scores_kernel<<<dim3((n_blocks + threads - 1) / threads, (unsigned)units), threads, 0,
                        (cudaStream_t)stream>>>(contrib, idx_c, n_kept, group, capacity, block,
                                                n_blocks, out);
  return launch_status();
}
