// E0 on tensor cores (bf16, head_dim 64/128): accumulated attention mass
//     s_j = sum_r softmax_j(q_r . K^T / sqrt(d))
// (Appendix B harness, H2O-style accumulated attention from observation
// queries) for one (batch row, KV head) unit per grid row.
//
// Pass 1, score_lse_mma_kernel: one CTA per (unit, block of 64 query rows);
// 4 warps x 16 rows.  Key tiles of 64 rows stream through a 2-stage TMA ring
// (128-byte swizzle); each warp computes S = Q K^T with mma.sync m16n8k16 and
// keeps a running (max, sum 2^(x - max)) per row; lse_r = max + log2(sum) in
// base 2, written to the workspace.
// Pass 2, score_col_mma_kernel: one CTA per (unit, block of 64 keys); the key
// tile is loaded once, the 4 warps walk the query rows 16 at a time and add
// 2^(x - lse_r) into per-lane column partials, which are reduced across
// lanes and warps in a fixed order (deterministic, no atomics).
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace ebd {

constexpr int kScTile = 64;     // keys per tile
constexpr int kScWarps = 4;
constexpr int kScRows = 16 * kScWarps;  // query rows per CTA in pass 1

template <int D>
struct ScoreLayout {
  static constexpr int kHalves = D / 64;
  static constexpr int kBoxBytes = kScTile * 128;          // 64 rows x 128 B
  static constexpr int kTileBytes = kHalves * kBoxBytes;   // one K tile
  static constexpr int kStages = 2;
  static constexpr int kBarOff = kStages * kTileBytes;
  static constexpr int kBytes = kBarOff + 2 * kStages * 8 + 1024;
};

// Byte offset of 16-byte chunk `chunk` (of the d dimension) of row `row` in a
// swizzled key tile: 64-column halves are separate boxes of 128-byte rows.
__device__ __forceinline__ uint32_t sw_off(int row, int chunk, int box_bytes) {
  return (uint32_t)((chunk >> 3) * box_bytes + row * 128 + (((chunk & 7) ^ (row & 7)) << 4));
}

// Q fragments (A operand, rows r0..r0+15 of the unit's observation queries)
// straight from global memory; rows >= R are zero.
template <int D>
__device__ __forceinline__ void load_q_frags(const __nv_bfloat16* Q, int R, int r0,
                                             uint32_t (&qa)[D / 16][4]) {
  const int lane = threadIdx.x & 31, g = lane >> 2, q = lane & 3;
  const int ra = r0 + g, rb = r0 + g + 8;
  const uint32_t* pa = reinterpret_cast<const uint32_t*>(Q + (size_t)(ra < R ? ra : 0) * D);
  const uint32_t* pb = reinterpret_cast<const uint32_t*>(Q + (size_t)(rb < R ? rb : 0) * D);
#pragma unroll
  for (int kk = 0; kk < D / 16; ++kk) {
    qa[kk][0] = ra < R ? __ldg(pa + 8 * kk + q) : 0u;
    qa[kk][1] = rb < R ? __ldg(pb + 8 * kk + q) : 0u;
    qa[kk][2] = ra < R ? __ldg(pa + 8 * kk + 4 + q) : 0u;
    qa[kk][3] = rb < R ? __ldg(pb + 8 * kk + 4 + q) : 0u;
  }
}

// S[16 x 64] = Qrows . Ktile^T for one warp: sc[nt][.] holds the C fragment
// of key columns 8nt .. 8nt+7.
template <int D>
__device__ __forceinline__ void qk_tile(const uint32_t (&qa)[D / 16][4], uint32_t kbase,
                                        float (&sc)[8][4]) {
  using L = ScoreLayout<D>;
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int nt = 0; nt < 8; ++nt) sc[nt][0] = sc[nt][1] = sc[nt][2] = sc[nt][3] = 0.f;
  // ldmatrix.x4: matrices (keys 16p..16p+7, chunk c), (.., c+1), (keys +8, c), (keys +8, c+1)
  const int krow = ((lane >> 4) << 3) + (lane & 7);
  const int csel = (lane >> 3) & 1;
#pragma unroll
  for (int kk = 0; kk < D / 16; ++kk) {
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      const int row = 16 * p + krow;
      uint32_t b0, b1, b2, b3;
      ldsm_x4(kbase + sw_off(row, 2 * kk + csel, L::kBoxBytes), b0, b1, b2, b3);
      mma_bf16_16816(sc[2 * p], qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3], b0, b1);
      mma_bf16_16816(sc[2 * p + 1], qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3], b2, b3);
    }
  }
}

template <int D>
__global__ void __launch_bounds__(kScWarps * 32) score_lse_mma_kernel(
    const __grid_constant__ CUtensorMap tmK, const __nv_bfloat16* __restrict__ q_obs, int n_ctx,
    int n_obs, float* __restrict__ lse, int32_t* dev_status) {
  using L = ScoreLayout<D>;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L::kBarOff);
  uint64_t* empty = full + L::kStages;
  const int unit = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r0 = blockIdx.y * kScRows + 16 * warp;
  const int tiles = (n_ctx + kScTile - 1) / kScTile;
  if (threadIdx.x == 0) {
    for (int s = 0; s < L::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kScWarps);
    }
    fence_barrier_init();
  }
  __syncthreads();
  const int key_row0 = unit * n_ctx;
  int issued = 0;  // meaningful in thread 0 only
  auto issue = [&](int t) {
    ++issued;
    const int s = t % L::kStages;
    unsigned char* st = smem + s * L::kTileBytes;
    mbar_arrive_expect_tx(&full[s], L::kTileBytes);
#pragma unroll
    for (int h = 0; h < L::kHalves; ++h)
      tma_load_2d(st + h * L::kBoxBytes, &tmK, h * 64, key_row0 + t * kScTile, &full[s]);
  };
  if (threadIdx.x == 0) {
    for (int t = 0; t < L::kStages && t < tiles; ++t) issue(t);
  }
  uint32_t qa[D / 16][4];
  load_q_frags<D>(q_obs + (size_t)unit * n_obs * D, n_obs, r0, qa);
  const float kscale = kLog2e * rsqrtf((float)D);
  const int q = lane & 3;
  float mrow[2] = {-INFINITY, -INFINITY}, srow[2] = {0.f, 0.f};
  bool ok = true;
  for (int t = 0; t < tiles; ++t) {
    const int s = t % L::kStages;
    if (!mbar_wait_bounded(&full[s], (uint32_t)((t / L::kStages) & 1))) {
      ok = false;
      break;
    }
    float sc[8][4];
    qk_tile<D>(qa, smem_u32(smem + s * L::kTileBytes), sc);
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[s]);
    if (threadIdx.x == 0 && t + L::kStages < tiles) {
      if (!mbar_wait_bounded(&empty[s], (uint32_t)((t / L::kStages) & 1))) {
        ok = false;
      } else {
        issue(t + L::kStages);
      }
    }
    const int kv = n_ctx - t * kScTile;  // valid keys in this tile
#pragma unroll
    for (int h = 0; h < 2; ++h) {  // rows g and g+8
      float mx = -INFINITY;
      float x[16];
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int col = 8 * nt + 2 * q + e;
          const float v = col < kv ? sc[nt][2 * h + e] * kscale : -INFINITY;
          x[2 * nt + e] = v;
          mx = fmaxf(mx, v);
        }
      }
      const float mn = fmaxf(mrow[h], mx);
      float acc = 0.f;
#pragma unroll
      for (int e = 0; e < 16; ++e) acc += exp2f(x[e] - mn);
      srow[h] = srow[h] * exp2f(mrow[h] - mn) + acc;
      mrow[h] = mn;
    }
  }
  if (threadIdx.x == 0) {  // never leave with copies in flight into shared memory
    for (int t = max(0, issued - L::kStages); t < issued; ++t)
      mbar_wait_bounded(&full[t % L::kStages], (uint32_t)((t / L::kStages) & 1));
  }
  if (!ok) {
    raise_status(dev_status, EBD_DEV_TIMEOUT);
    return;
  }
  // combine the 4 lanes of each row
#pragma unroll
  for (int h = 0; h < 2; ++h) {
#pragma unroll
    for (int o = 1; o <= 2; o <<= 1) {
      const float mo = __shfl_xor_sync(0xffffffffu, mrow[h], o);
      const float so = __shfl_xor_sync(0xffffffffu, srow[h], o);
      const float mn = fmaxf(mrow[h], mo);
      srow[h] = (mrow[h] == -INFINITY ? 0.f : srow[h] * exp2f(mrow[h] - mn)) +
                (mo == -INFINITY ? 0.f : so * exp2f(mo - mn));
      mrow[h] = mn;
    }
  }
  if (q == 0) {
    const int g = lane >> 2;
    if (r0 + g < n_obs) lse[(size_t)unit * n_obs + r0 + g] = mrow[0] + log2f(srow[0]);
    if (r0 + g + 8 < n_obs) lse[(size_t)unit * n_obs + r0 + g + 8] = mrow[1] + log2f(srow[1]);
  }
}

template <int D>
__global__ void __launch_bounds__(kScWarps * 32) score_col_mma_kernel(
    const __grid_constant__ CUtensorMap tmK, const __nv_bfloat16* __restrict__ q_obs, int n_ctx,
    int n_obs, const float* __restrict__ lse, float* __restrict__ scores, int32_t* dev_status) {
  using L = ScoreLayout<D>;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L::kBarOff);
  __shared__ float colsum[kScWarps][kScTile];
  const int unit = blockIdx.x, kt = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, q = lane & 3;
  if (threadIdx.x == 0) {
    mbar_init(&full[0], 1);
    fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    mbar_arrive_expect_tx(&full[0], L::kTileBytes);
#pragma unroll
    for (int h = 0; h < L::kHalves; ++h)
      tma_load_2d(smem + h * L::kBoxBytes, &tmK, h * 64, unit * n_ctx + kt * kScTile, &full[0]);
  }
  const float kscale = kLog2e * rsqrtf((float)D);
  const int kv = n_ctx - kt * kScTile;
  float part[8][2];
#pragma unroll
  for (int nt = 0; nt < 8; ++nt) part[nt][0] = part[nt][1] = 0.f;
  const bool ok = mbar_wait_bounded(&full[0], 0u);
  if (ok) {
    const __nv_bfloat16* Qu = q_obs + (size_t)unit * n_obs * D;
    const float* lu = lse + (size_t)unit * n_obs;
    const uint32_t kbase = smem_u32(smem);
    for (int r0 = 16 * warp; r0 < n_obs; r0 += 16 * kScWarps) {
      uint32_t qa[D / 16][4];
      load_q_frags<D>(Qu, n_obs, r0, qa);
      float sc[8][4];
      qk_tile<D>(qa, kbase, sc);
      const float la = r0 + g < n_obs ? __ldg(lu + r0 + g) : INFINITY;
      const float lb = r0 + g + 8 < n_obs ? __ldg(lu + r0 + g + 8) : INFINITY;
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          part[nt][e] += exp2f(fmaf(sc[nt][e], kscale, -la)) + exp2f(fmaf(sc[nt][2 + e], kscale, -lb));
        }
      }
    }
  } else {
    raise_status(dev_status, EBD_DEV_TIMEOUT);
  }
  // reduce over the 8 row groups of the warp, then over the warps, in a fixed order
#pragma unroll
  for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      float v = part[nt][e];
      v += __shfl_xor_sync(0xffffffffu, v, 4);
      v += __shfl_xor_sync(0xffffffffu, v, 8);
      v += __shfl_xor_sync(0xffffffffu, v, 16);
      if (g == 0) colsum[warp][8 * nt + 2 * q + e] = v;
    }
  }
  __syncthreads();
  for (int c = threadIdx.x; c < kScTile; c += kScWarps * 32) {
    float v = 0.f;
#pragma unroll
    for (int w = 0; w < kScWarps; ++w) v += colsum[w][c];
    if (c < kv) scores[(size_t)unit * n_ctx + kt * kScTile + c] = v;
  }
}

static PFN_cuTensorMapEncodeTiled_v12000 score_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

template <int D>
static ebd_status launch_score_mma_t(int units, int n_ctx, int n_obs, const void* q_obs,
                                     const void* K, float* scores, float* lse,
                                     int32_t* dev_status, cudaStream_t s) {
  using L = ScoreLayout<D>;
  auto enc = score_encoder();
  if (!enc) return EBD_ERR_CUDA;
  CUtensorMap tmK;
  const cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)units * n_ctx};
  const cuuint64_t strides[1] = {(cuuint64_t)D * 2};
  const cuuint32_t box[2] = {64, (cuuint32_t)kScTile};
  const cuuint32_t estr[2] = {1, 1};
  if (enc(&tmK, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(K), dims, strides, box, estr,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return EBD_ERR_CUDA;
  const int smem = L::kBytes;
  if (cudaFuncSetAttribute(score_lse_mma_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           smem) != cudaSuccess ||
      cudaFuncSetAttribute(score_col_mma_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           smem) != cudaSuccess)
    return EBD_ERR_CUDA;
  const __nv_bfloat16* Q = reinterpret_cast<const __nv_bfloat16*>(q_obs);
  dim3 g1(units, (n_obs + kScRows - 1) / kScRows);
  score_lse_mma_kernel<D><<<g1, kScWarps * 32, smem, s>>>(tmK, Q, n_ctx, n_obs, lse, dev_status);
  ebd_status st = launch_status();
  if (st != EBD_OK) return st;
  dim3 g2(units, (n_ctx + kScTile - 1) / kScTile);
  score_col_mma_kernel<D><<<g2, kScWarps * 32, smem, s>>>(tmK, Q, n_ctx, n_obs, lse, scores,
                                                          dev_status);
  return launch_status();
}

bool score_mma_supported(ebd_dtype dtype, int head_dim, const void* q_obs, const void* K) {
  return dtype == EBD_BF16 && (head_dim == 64 || head_dim == 128) &&
         ((uintptr_t)q_obs & 15u) == 0 && ((uintptr_t)K & 15u) == 0 && score_encoder() != nullptr;
}

ebd_status launch_score_mma(int units, int head_dim, int n_ctx, int n_obs, const void* q_obs,
                            const void* K, float* scores, float* lse, int32_t* dev_status,
                            cudaStream_t s) {
  if ((long long)units * n_ctx >= 0x7fffffffLL) return EBD_ERR_UNSUPPORTED;
  if (head_dim == 128)
    return launch_score_mma_t<128>(units, n_ctx, n_obs, q_obs, K, scores, lse, dev_status, s);
  if (head_dim == 64)
    return launch_score_mma_t<64>(units, n_ctx, n_obs, q_obs, K, scores, lse, dev_status, s);
  return EBD_ERR_UNSUPPORTED;
}

}  // namespace ebd
