// Tensor-core certified decode (bf16 compact cache, head_dim 64/128, G <= 8).
//
// Same quantities as the CUDA-core path (Eq. 3, Theorem 2, Eq. 4): per query
// head an online softmax over logits q.k/sqrt(d) + log(1/pi) carrying
// l = sum w, o = sum w v, U = sum u, A1 = sum u v, A2 = sum u ||v||^2 and the
// range-bound maxima, with u = (1 - pi) w^2.
//
// Layout of the work.  A persistent grid (one CTA per SM) of 8 warps.  The
// active 16-token tiles of all units (tiles
// below min(n_kept, cap), counted by a one-CTA plan kernel into tile_off) are
// split into equal contiguous ranges, one per warp.  A warp's range
// crosses at most a few units; for each unit it meets it writes one partial
// record, at index (unit + global warp), so records never collide and no
// scratch needs clearing.  The reduce kernel merges the records of a unit.
//
// Per tile and warp:
//   S[16 x 16]  = Qpad[16 x d] . K_tile^T       (rows 0..G-1 = query heads,
//                                                rows 8..15 = 0; 2 x d/16 mma)
//   w = 2^(S log2e/sqrt(d) + log2e log(1/pi) - M), u = (1 - pi) w^2
//   P[16 x 16]  = [w (rows 0..7); u (rows 8..15)] as bf16 hi + bf16 lo parts
//   acc[16 x d] += P_hi . V_tile + P_lo . V_tile   (rows 0..7: o, rows 8..15: A1)
// The hi/lo split keeps ~16 mantissa bits of the weights on bf16 tensor
// cores.  ||v||^2 per token comes from the same V fragments (squares summed
// over the lanes that hold one token).  The running maximum is updated
// lazily: accumulators are rescaled only when a row's maximum grows by more
// than 2^8, so weights stay below 2^8 and u below 2^16.
//
// Each warp streams its own tiles: one lane issues the 2D TMA copies (128-byte
// swizzle) of K and V and a 64-byte bulk copy of log(1/pi) for tile j + 2 into
// its private 3-stage ring while tile j is consumed; every stage has one
// transaction-counting mbarrier.  A stage is refilled only after the same warp
// has read it (ordered by a proxy fence), so no empty barrier is needed.
// Every wait is bounded (~2 s); on timeout the kernel raises EBD_DEV_TIMEOUT,
// drains the copies it issued and returns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "decode.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace ebd {

constexpr int kMmaTile = 16;
constexpr int kMmaConsumers = 8;  // warps per CTA
constexpr int kMmaStagesPerWarp = 3;
constexpr int kMmaStages = kMmaConsumers * kMmaStagesPerWarp;
constexpr int kMmaThreads = kMmaConsumers * 32;
constexpr float kRescaleLog2 = 8.f;
constexpr int kMinTilesPerWarp = 4;

template <int D>
struct MmaLayout {
  static constexpr int kHalves = D / 64;                 // 64-column TMA boxes per row
  static constexpr int kBoxBytes = kMmaTile * 128;      // one box: 16 rows x 128 B
  static constexpr int kStageBytes = 2 * kHalves * kBoxBytes;
  static constexpr int kLogwOff = kMmaStages * kStageBytes;
  static constexpr int kBarOff = kLogwOff + kMmaStages * kMmaTile * 4;
  static constexpr int kBytes = kBarOff + kMmaStages * 8 + 1024;  // + alignment slack
  static constexpr uint32_t kTxBytes = 2 * kHalves * kBoxBytes + kMmaTile * 4;
};

struct FastArgs {
  const __nv_bfloat16* Q;  // [units * G, D]
  const float* logw;       // [units, cap]
  const int32_t* n_kept;   // [units]
  const int32_t* tile_off;  // [units + 1], written by the plan kernel
  float* part;             // records [(units + W) * G, rec_floats(D)]
  int32_t* dev_status;
  int units;
  int cap;
  int group;
};

// Largest unit u with tile_off[u] <= t (a unit that holds tile t).
__device__ __forceinline__ int unit_of_tile(const int32_t* tile_off, int units, int t) {
  int lo = 0, hi = units - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (__ldg(tile_off + mid) <= t) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// Next unit after u that holds at least one tile (tile t exists beyond u).
__device__ __forceinline__ int next_unit(const int32_t* tile_off, int u) {
  ++u;
  while (__ldg(tile_off + u + 1) == __ldg(tile_off + u)) ++u;
  return u;
}

// Exclusive prefix of active (16-token) tiles per unit: tile_off[u], with
// tile_off[units] = the total.
__global__ void decode_tile_plan_kernel(const int32_t* __restrict__ n_kept, int units, int cap,
                                        int32_t* __restrict__ tile_off) {
  __shared__ int warp_tot[32];
  __shared__ int carry;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) carry = 0;
  __syncthreads();
  for (int base = 0; base < units; base += blockDim.x) {
    const int u = base + tid;
    const int v = u < units ? (min(max(n_kept[u], 0), cap) + kMmaTile - 1) / kMmaTile : 0;
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int n = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += n;
    }
    if (lane == 31) warp_tot[warp] = incl;
    __syncthreads();
    if (warp == 0) {
      const int nw = blockDim.x >> 5;
      const int x = lane < nw ? warp_tot[lane] : 0;
      int wi = x;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int n = __shfl_up_sync(0xffffffffu, wi, o);
        if (lane >= o) wi += n;
      }
      if (lane < nw) warp_tot[lane] = wi - x;
    }
    __syncthreads();
    const int excl = carry + warp_tot[warp] + incl - v;
    if (u < units) tile_off[u] = excl;
    __syncthreads();
    if (tid == blockDim.x - 1) carry = excl + v;
    __syncthreads();
  }
  if (tid == 0) tile_off[units] = carry;
}

template <int D>
__global__ void __launch_bounds__(kMmaThreads, 1)
    decode_mma_kernel(const __grid_constant__ CUtensorMap tmK,
                      const __grid_constant__ CUtensorMap tmV, FastArgs a) {
  using L = MmaLayout<D>;
  constexpr int REC = rec_floats(D);
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem =
      (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);  // swizzle atoms
  float* lw_s = reinterpret_cast<float*>(smem + L::kLogwOff);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L::kBarOff);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kMmaStages; ++s) mbar_init(&full[s], 1);
    fence_barrier_init();
  }
  __syncthreads();

  const int units = a.units;
  const int Ta = __ldg(a.tile_off + units);
  if (Ta == 0) return;
  const long long Wall = (long long)gridDim.x * kMmaConsumers;
  // working warps: every one gets >= kMinTilesPerWarp tiles (bounded merge work)
  const long long Wcap = Ta / kMinTilesPerWarp > 0 ? Ta / kMinTilesPerWarp : 1;
  const long long W = Wall < Wcap ? Wall : Wcap;

  // global warp index, consecutive indices on different SMs
  const long long gw = (long long)warp * gridDim.x + blockIdx.x;
  if (gw >= W) return;
  const int tb = (int)(gw * Ta / W);
  const int te = (int)((gw + 1) * Ta / W);
  const int G = a.group;
  const int g = lane >> 2, q = lane & 3;
  const float kscale = kLog2e * rsqrtf((float)D);
  uint64_t* my_full = full + warp * kMmaStagesPerWarp;

  // copies: lane 0 walks its own cursor through the warp's tiles
  int pf_t = tb, pf_u = unit_of_tile(a.tile_off, units, tb);
  int pf_lo = __ldg(a.tile_off + pf_u), pf_hi = __ldg(a.tile_off + pf_u + 1);
  int issued = 0;
  auto issue_next = [&]() {
    if (lane == 0 && pf_t < te) {
      const int s = issued % kMmaStagesPerWarp;
      const int stage = warp * kMmaStagesPerWarp + s;
      const int row0 = pf_u * a.cap + (pf_t - pf_lo) * kMmaTile;
      unsigned char* st = smem + (size_t)stage * L::kStageBytes;
      mbar_arrive_expect_tx(&my_full[s], L::kTxBytes);
#pragma unroll
      for (int h = 0; h < L::kHalves; ++h) {
        tma_load_2d(st + h * L::kBoxBytes, &tmK, h * 64, row0, &my_full[s]);
        tma_load_2d(st + (L::kHalves + h) * L::kBoxBytes, &tmV, h * 64, row0, &my_full[s]);
      }
      bulk_load(lw_s + stage * kMmaTile, a.logw + row0, kMmaTile * 4, &my_full[s]);
      ++pf_t;
      if (pf_t < te && pf_t == pf_hi) {
        pf_u = next_unit(a.tile_off, pf_u);
        pf_lo = pf_hi;
        pf_hi = __ldg(a.tile_off + pf_u + 1);
      }
    }
    ++issued;
  };

  float acc[D / 8][4];
  float M2 = -INFINITY, l = 0.f, U = 0.f, A2 = 0.f, cmax = 0.f, umax = 0.f;
  uint32_t qa[D / 16][2];
  int u = pf_u;
  int seg_end = 0, n_u = 0, seg_start = 0;

  auto begin_segment = [&]() {
    seg_start = __ldg(a.tile_off + u);
    seg_end = __ldg(a.tile_off + u + 1);
    n_u = min(__ldg(a.n_kept + u), a.cap);
    const uint32_t* qrow =
        reinterpret_cast<const uint32_t*>(a.Q + ((size_t)u * G + (g < G ? g : 0)) * D);
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      qa[kk][0] = g < G ? __ldg(qrow + 8 * kk + q) : 0u;
      qa[kk][1] = g < G ? __ldg(qrow + 8 * kk + 4 + q) : 0u;
    }
#pragma unroll
    for (int j = 0; j < D / 8; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;
    M2 = -INFINITY;
    l = U = A2 = cmax = umax = 0.f;
  };

  auto flush_segment = [&]() {
#pragma unroll
    for (int o = 1; o <= 2; o <<= 1) {
      l += __shfl_xor_sync(0xffffffffu, l, o);
      U += __shfl_xor_sync(0xffffffffu, U, o);
      A2 += __shfl_xor_sync(0xffffffffu, A2, o);
      cmax = fmaxf(cmax, __shfl_xor_sync(0xffffffffu, cmax, o));
      umax = fmaxf(umax, __shfl_xor_sync(0xffffffffu, umax, o));
    }
    if (g < G) {
      float* rec = a.part + ((size_t)(u + gw) * G + g) * REC;
      if (q == 0) {
        rec[kRecM] = M2 == -INFINITY ? -INFINITY : M2 * kLn2;
        rec[kRecL] = l;
        rec[kRecU] = U;
        rec[kRecA2] = A2;
        rec[kRecCmax] = cmax;
        rec[kRecUmax] = umax;
      }
#pragma unroll
      for (int j = 0; j < D / 8; ++j) {
        *reinterpret_cast<float2*>(rec + kRecHead + 8 * j + 2 * q) = make_float2(acc[j][0], acc[j][1]);
        *reinterpret_cast<float2*>(rec + kRecHead + D + 8 * j + 2 * q) =
            make_float2(acc[j][2], acc[j][3]);
      }
    }
  };

  // prologue: the first stages of the ring
#pragma unroll
  for (int p = 0; p < kMmaStagesPerWarp - 1; ++p) issue_next();

  begin_segment();
  bool ok = true;
  int j = 0;
  for (int t = tb; t < te; ++t, ++j) {
    issue_next();  // tile j + 2 into the stage tile j - 1 left
    if (t == seg_end) {
      flush_segment();
      u = next_unit(a.tile_off, u);
      begin_segment();
    }
    const int n_valid = min(kMmaTile, n_u - (t - seg_start) * kMmaTile);
    const int sl = j % kMmaStagesPerWarp;
    const int s = warp * kMmaStagesPerWarp + sl;
    if (!mbar_wait_bounded(&my_full[sl], (uint32_t)((j / kMmaStagesPerWarp) & 1))) {
      ok = false;
      break;
    }
    const uint32_t kbase = smem_u32(smem + (size_t)s * L::kStageBytes);
    const uint32_t vbase = kbase + L::kHalves * L::kBoxBytes;

    // ---- S = Q K^T ---------------------------------------------------------
    float sc0[4] = {0.f, 0.f, 0.f, 0.f}, sc1[4] = {0.f, 0.f, 0.f, 0.f};
    {
      const int tok = ((lane >> 4) << 3) + (lane & 7);
      const int half_sel = (lane >> 3) & 1;
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const int chunk = 2 * kk + half_sel;
        const uint32_t addr = kbase + (chunk >> 3) * L::kBoxBytes + tok * 128 +
                              (((chunk & 7) ^ (tok & 7)) << 4);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(addr, b0, b1, b2, b3);
        mma_bf16_16816(sc0, qa[kk][0], 0u, qa[kk][1], 0u, b0, b1);
        mma_bf16_16816(sc1, qa[kk][0], 0u, qa[kk][1], 0u, b2, b3);
      }
    }

    // ---- weights -----------------------------------------------------------
    const float2 lwa = *reinterpret_cast<const float2*>(lw_s + s * kMmaTile + 2 * q);
    const float2 lwb = *reinterpret_cast<const float2*>(lw_s + s * kMmaTile + 8 + 2 * q);
    const float lwv[4] = {lwa.x, lwa.y, lwb.x, lwb.y};
    const int tk[4] = {2 * q, 2 * q + 1, 8 + 2 * q, 9 + 2 * q};
    const float sv[4] = {sc0[0], sc0[1], sc1[0], sc1[1]};
    float x[4];
    float mx = -INFINITY;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      x[i] = tk[i] < n_valid ? fmaf(sv[i], kscale, lwv[i] * kLog2e) : -INFINITY;
      mx = fmaxf(mx, x[i]);
    }
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
    if (mx > M2 + kRescaleLog2) {
      const float f = exp2f(M2 - mx), f2 = f * f;
#pragma unroll
      for (int jj = 0; jj < D / 8; ++jj) {
        acc[jj][0] *= f;
        acc[jj][1] *= f;
        acc[jj][2] *= f2;
        acc[jj][3] *= f2;
      }
      l *= f;
      U *= f2;
      A2 *= f2;
      cmax *= f;
      umax *= f;
      M2 = mx;
    }
    float wv[4], uv[4], suv[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const bool val = tk[i] < n_valid;
      wv[i] = exp2f(x[i] - M2);
      const float omp = val ? one_minus_exp_neg(lwv[i]) : 0.f;  // 1 - pi
      uv[i] = omp * wv[i] * wv[i];
      suv[i] = sqrtf(omp) * wv[i];
      umax = fmaxf(umax, suv[i]);
    }
    const uint32_t h0 = pack_bf16(wv[0], wv[1]), h1 = pack_bf16(uv[0], uv[1]);
    const uint32_t h2 = pack_bf16(wv[2], wv[3]), h3 = pack_bf16(uv[2], uv[3]);
    const uint32_t r0 = pack_bf16(wv[0] - bf16_lo(h0), wv[1] - bf16_hi(h0));
    const uint32_t r1 = pack_bf16(uv[0] - bf16_lo(h1), uv[1] - bf16_hi(h1));
    const uint32_t r2 = pack_bf16(wv[2] - bf16_lo(h2), wv[3] - bf16_hi(h2));
    const uint32_t r3 = pack_bf16(uv[2] - bf16_lo(h3), uv[3] - bf16_hi(h3));
    // The scalar sums use exactly the weights the tensor cores multiply with
    // (hi + lo), so that V_hat = (A2 - 2 y.A1 + |y|^2 U) / l^2 cancels
    // consistently when y_hat sits close to the retained values.
    const float wt[4] = {bf16_lo(h0) + bf16_lo(r0), bf16_hi(h0) + bf16_hi(r0),
                         bf16_lo(h2) + bf16_lo(r2), bf16_hi(h2) + bf16_hi(r2)};
    const float ut[4] = {bf16_lo(h1) + bf16_lo(r1), bf16_hi(h1) + bf16_hi(r1),
                         bf16_lo(h3) + bf16_lo(r3), bf16_hi(h3) + bf16_hi(r3)};
    l += (wt[0] + wt[1]) + (wt[2] + wt[3]);
    U += (ut[0] + ut[1]) + (ut[2] + ut[3]);

    // ---- acc += P V, ||v||^2 -------------------------------------------------
    const uint32_t m01 = (tk[0] < n_valid ? 0x0000ffffu : 0u) | (tk[1] < n_valid ? 0xffff0000u : 0u);
    const uint32_t m23 = (tk[2] < n_valid ? 0x0000ffffu : 0u) | (tk[3] < n_valid ? 0xffff0000u : 0u);
    float2 vn01 = make_float2(0.f, 0.f), vn23 = make_float2(0.f, 0.f);
    {
      const int tok = ((lane >> 3) & 1) * 8 + (lane & 7);
      const int chunk_sel = lane >> 4;
#pragma unroll
      for (int jp = 0; jp < D / 16; ++jp) {
        const int chunk = 2 * jp + chunk_sel;
        const uint32_t addr = vbase + (chunk >> 3) * L::kBoxBytes + tok * 128 +
                              (((chunk & 7) ^ (tok & 7)) << 4);
        uint32_t v0, v1, v2, v3;
        ldsm_x4_trans(addr, v0, v1, v2, v3);
        v0 &= m01;
        v2 &= m01;
        v1 &= m23;
        v3 &= m23;
        const float2 f0 = make_float2(bf16_lo(v0), bf16_hi(v0));
        const float2 f1 = make_float2(bf16_lo(v1), bf16_hi(v1));
        const float2 f2 = make_float2(bf16_lo(v2), bf16_hi(v2));
        const float2 f3 = make_float2(bf16_lo(v3), bf16_hi(v3));
        vn01 = __ffma2_rn(f0, f0, __ffma2_rn(f2, f2, vn01));
        vn23 = __ffma2_rn(f1, f1, __ffma2_rn(f3, f3, vn23));
        mma_bf16_16816(acc[2 * jp], h0, h1, h2, h3, v0, v1);
        mma_bf16_16816(acc[2 * jp], r0, r1, r2, r3, v0, v1);
        mma_bf16_16816(acc[2 * jp + 1], h0, h1, h2, h3, v2, v3);
        mma_bf16_16816(acc[2 * jp + 1], r0, r1, r2, r3, v2, v3);
      }
    }
    // reads of this stage are done before a later copy overwrites it
    fence_proxy_async_smem();
    __syncwarp();
    float vn[4] = {vn01.x, vn01.y, vn23.x, vn23.y};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      vn[i] += __shfl_xor_sync(0xffffffffu, vn[i], 4);
      vn[i] += __shfl_xor_sync(0xffffffffu, vn[i], 8);
      vn[i] += __shfl_xor_sync(0xffffffffu, vn[i], 16);
      A2 = fmaf(ut[i], vn[i], A2);
      cmax = fmaxf(cmax, suv[i] * sqrtf(vn[i]));
    }
  }
  if (!ok) raise_status(a.dev_status, EBD_DEV_TIMEOUT);
  else flush_segment();
  // never leave with copies in flight into this CTA's shared memory
  if (lane == 0) {
    const int n_iss = min(issued, te - tb);
#pragma unroll 1
    for (int k = max(0, n_iss - kMmaStagesPerWarp); k < n_iss; ++k)
      mbar_wait_bounded(&my_full[k % kMmaStagesPerWarp], (uint32_t)((k / kMmaStagesPerWarp) & 1));
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
static PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
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

// [rows, D] bf16 viewed as 2D; box = 64 columns x 16 rows, 128-byte swizzle.
static bool encode_rows_map(CUtensorMap* map, const void* base, long long rows, int D) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)D * 2};
  const cuuint32_t box[2] = {64, (cuuint32_t)kMmaTile};
  const cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool fast_decode_supported(ebd_dtype dtype, int group, int head_dim, int capacity) {
  return dtype == EBD_BF16 && (head_dim == 64 || head_dim == 128) && group >= 1 && group <= 8 &&
         capacity % kMmaTile == 0;
}

void fast_decode_plan(DecodePlan& p, long long units, int group, int head_dim, int capacity) {
  (void)capacity;
  p.ctas = sm_count();
  const long long W = (long long)p.ctas * kMmaConsumers;
  p.ws_bytes = fast_decode_records_offset((int)units) +
               align_up((size_t)(units + W) * group * rec_floats(head_dim) * sizeof(float), 256);
}

static bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

long long fast_decode_warps(const DecodePlan& p) { return (long long)p.ctas * kMmaConsumers; }

int fast_decode_min_tiles_per_warp() { return kMinTilesPerWarp; }

// Workspace: tile_off [units + 1] | records.
size_t fast_decode_records_offset(int units) {
  return align_up((size_t)(units + 1) * sizeof(int32_t), 256);
}

bool fast_decode_usable(const DecodeArgs& a, int units) {
  return aligned16(a.Kc) && aligned16(a.Vc) && aligned16(a.logw) && aligned16(a.Q) &&
         (long long)units * a.cap < 0x7fffffffLL && tensor_map_encoder() != nullptr;
}

template <int D>
static ebd_status launch_fast_t(const DecodePlan& plan, const DecodeArgs& a, int units,
                                cudaStream_t s) {
  CUtensorMap tmK, tmV;
  const long long rows = (long long)units * a.cap;
  if (!encode_rows_map(&tmK, a.Kc, rows, D) || !encode_rows_map(&tmV, a.Vc, rows, D))
    return EBD_ERR_CUDA;
  int32_t* tile_off = reinterpret_cast<int32_t*>(a.part);
  float* recs = reinterpret_cast<float*>(reinterpret_cast<char*>(a.part) +
                                         fast_decode_records_offset(units));
  decode_tile_plan_kernel<<<1, 1024, 0, s>>>(a.n_kept, units, a.cap, tile_off);
  ebd_status st = launch_status();
  if (st != EBD_OK) return st;
  FastArgs f;
  f.Q = reinterpret_cast<const __nv_bfloat16*>(a.Q);
  f.logw = a.logw;
  f.n_kept = a.n_kept;
  f.tile_off = tile_off;
  f.part = recs;
  f.dev_status = a.dev_status;
  f.units = units;
  f.cap = a.cap;
  f.group = a.group;
  const int smem = MmaLayout<D>::kBytes;
  if (cudaFuncSetAttribute(decode_mma_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           smem) != cudaSuccess)
    return EBD_ERR_CUDA;
  decode_mma_kernel<D><<<plan.ctas, kMmaThreads, smem, s>>>(tmK, tmV, f);
  return launch_status();
}

ebd_status launch_fast_decode(ebd_dtype dtype, int head_dim, const DecodePlan& plan,
                              const DecodeArgs& a, int units, cudaStream_t stream) {
  if (dtype != EBD_BF16) return EBD_ERR_UNSUPPORTED;
  if (head_dim == 128) return launch_fast_t<128>(plan, a, units, stream);
  if (head_dim == 64) return launch_fast_t<64>(plan, a, units, stream);
  return EBD_ERR_UNSUPPORTED;
}

}  // namespace ebd
