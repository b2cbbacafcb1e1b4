// E0 on the 5th-generation tensor cores: accumulated attention mass
//     s_j = sum_r softmax_j(q_r . K^T / sqrt(d))
// (Appendix B harness, H2O-style accumulated attention from R observation
// query rows of a KV head's group), bf16 inputs, f32 accumulation in tensor
// memory, head_dim 64/128, R <= 512.
//
// Pass 1, score_lse_tc_kernel: one CTA per (unit, 128 query rows).  The rows
// are the MMA's M (= tensor-memory lanes), 256-key tiles its N, so the
// accumulator S[128 x 256] = Q K^T holds one query row per lane and the
// epilogue thread that owns a lane keeps that row's running
// (max, sum 2^(x - max)) without any cross-thread traffic.  Two accumulators
// (256 columns each) alternate so the MMA of tile j + 1 overlaps the epilogue
// of tile j; three shared-memory stages of K let the copy of tile j + 2 start
// when the MMA of tile j - 1 is done.  Output: the base-2 log-sum-exp of
// every row (workspace).
// Pass 2, score_col_tc_kernel: the transposed product S^T = K Q^T, keys as M
// (one key per lane), all R query rows as N (split in two halves of <= 256
// columns, one per accumulator), so key j's thread sums 2^(x_rj - lse_r) over
// its own row.  A persistent grid walks (unit, 128-key tile) items in order,
// reloading Q only when the unit changes.
//
// Roles: warps 0-15 are the epilogue (warps w, w + 4, w + 8, w + 12 read
// tensor-memory lanes 32 (w % 4) .. + 31; in pass 1 warp w takes the 64
// columns from 64 (w / 4) on, in pass 2 every fourth 32-column chunk of the
// accumulator); warp 16 allocates tensor memory and one of its lanes
// issues the TMA copies (128-byte swizzle) and the tcgen05.mma instructions.
// Hand-offs use mbarriers: TMA -> MMA (transaction counts), MMA -> epilogue
// and MMA -> smem reuse (tcgen05.commit), epilogue -> MMA (512 arrivals).  The
// four warps of a lane quarter combine their parts of a row (pass 1) or of a
// key's sum (pass 2) through shared memory, in a fixed order.
// Every wait is bounded (~2 s); a timeout raises EBD_DEV_TIMEOUT, the roles
// leave their loops and the tensor memory is released.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "internal.h"
#include "ptx.cuh"
#include "tcgen05.cuh"

namespace ebd {

constexpr int kTcRows1 = 128;   // pass 1: query rows per CTA (MMA M)
constexpr int kTcKeys1 = 256;   // pass 1: keys per tile (MMA N)
constexpr int kTcKeys2 = 128;   // pass 2: keys per tile (MMA M)
constexpr int kTcMaxRows = 512; // pass 2: query rows held as accumulator columns
constexpr int kTcGroups = 4;    // epilogue warps per tensor-memory lane quarter
constexpr int kTcEpi = 128 * kTcGroups;  // epilogue threads
constexpr int kTcThreads = kTcEpi + 32;  // + 1 issue warp
constexpr int kTcIssueWarp = kTcEpi / 32;
constexpr uint32_t kTmemCols = 512;

template <int D>
struct Tc1Layout {
  static constexpr int kHalves = D / 64;             // 64-column (128-byte) boxes
  static constexpr int kQBox = kTcRows1 * 128;       // 16 KB
  static constexpr int kKBox = kTcKeys1 * 128;       // 32 KB
  static constexpr int kKOff = kHalves * kQBox;
  static constexpr int kStages = 3;                  // K tiles in flight
  static constexpr int kBarOff = kKOff + kStages * kHalves * kKBox;
  // [groups][128][2] f32 of the final combine, over the K stages (all MMAs
  // have completed by then)
  static constexpr int kPartOff = kKOff;
  static constexpr int kBytes = kBarOff + 16 * 8 + 1024;  // + alignment slack
};

template <int D>
struct Tc2Layout {
  static constexpr int kHalves = D / 64;
  static constexpr int kQBox = kTcMaxRows * 128;     // 64 KB (rows beyond R unused)
  static constexpr int kKBox = kTcKeys2 * 128;       // 16 KB
  static constexpr int kKOff = kHalves * kQBox;
  static constexpr int kLseOff = kKOff + 2 * kHalves * kKBox;  // [2][kTcMaxRows] f32
  static constexpr int kPartOff = kLseOff + 2 * kTcMaxRows * 4;  // [2][groups][128] f32
  static constexpr int kBarOff = kPartOff + 2 * kTcGroups * 128 * 4;
  static constexpr int kBytes = kBarOff + 16 * 8 + 1024;
};

struct TcArgs {
  int units;
  int n_ctx;     // N
  int n_obs;     // R
  int mtiles;    // pass 1: ceil(R / 128)
  int rows_pad;  // pass 2: R rounded up to 32
  int n_a;       // pass 2: accumulator A columns (<= 256)
  int n_b;       // pass 2: accumulator B columns (rows_pad - n_a)
  int items;     // pass 2: units * ceil(N / 128)
  float scale2;  // log2(e) / sqrt(d)
  float* lse2;   // [units, R] base-2 log-sum-exp (pass 1 out, pass 2 in)
  float* scores; // [units, N]
  int32_t* dev_status;
};

// max(a, b, c) in one instruction (three-input form of max.f32).
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

__device__ __forceinline__ unsigned char* align1024(unsigned char* p) {
  return (unsigned char*)(((uintptr_t)p + 1023) & ~(uintptr_t)1023);
}

template <int D>
__global__ void __launch_bounds__(kTcThreads, 1)
    score_lse_tc_kernel(const __grid_constant__ CUtensorMap tmQ,
                        const __grid_constant__ CUtensorMap tmK, TcArgs a) {
  using L = Tc1Layout<D>;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = align1024(smem_raw);
  constexpr int KS = L::kStages;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::kBarOff);
  uint64_t* q_full = bars;
  uint64_t* k_full = bars + 1;          // [KS]
  uint64_t* k_empty = k_full + KS;      // [KS]
  uint64_t* acc_full = k_empty + KS;    // [2]
  uint64_t* acc_empty = acc_full + 2;   // [2]
  uint64_t* mma_done = acc_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int unit = blockIdx.x / a.mtiles, mt = blockIdx.x - unit * a.mtiles;
  const int nk = (a.n_ctx + kTcKeys1 - 1) / kTcKeys1;
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < KS; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&acc_full[s], 1);
      mbar_init(&acc_empty[s], kTcEpi);
    }
    mbar_init(mma_done, 1);
    fence_barrier_init();
  }
  if (warp == kTcIssueWarp) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  bool ok = true;
  const int quarter = warp & 3, grp = warp >> 2;  // epilogue lane quarter, chunk group
  const int row = quarter * 32 + lane;
  float m = -INFINITY, ssum = 0.f;  // epilogue: raw max logit and sum 2^((x - m) scale2)

  if (warp == kTcIssueWarp) {
    if (lane == 0) {
      const int krow0 = unit * a.n_ctx;
      mbar_arrive_expect_tx(q_full, L::kHalves * L::kQBox);
#pragma unroll
      for (int h = 0; h < L::kHalves; ++h)
        tma_load_2d(smem + h * L::kQBox, &tmQ, h * 64, unit * a.n_obs + mt * kTcRows1, q_full);
      auto load_k = [&](int j) {
        const int s = j % KS;
        mbar_arrive_expect_tx(&k_full[s], L::kHalves * L::kKBox);
#pragma unroll
        for (int h = 0; h < L::kHalves; ++h)
          tma_load_2d(smem + L::kKOff + (s * L::kHalves + h) * L::kKBox, &tmK, h * 64,
                      krow0 + j * kTcKeys1, &k_full[s]);
      };
      int issued = 0, consumed = 0;
      for (; issued < nk && issued < KS; ++issued) load_k(issued);
      const bool q_ok = mbar_wait_bounded(q_full, 0);
      ok = q_ok;
      const uint32_t idesc = umma_idesc_bf16_f32(128, kTcKeys1);
      const uint32_t qbase = smem_u32(smem);
      for (int j = 0; ok && j < nk; ++j) {
        const int s = j % KS, b = j & 1;  // K stage, accumulator
        if (!mbar_wait_bounded(&k_full[s], (j / KS) & 1)) {
          ok = false;
          break;
        }
        ++consumed;
        if (j >= 2 && !mbar_wait_bounded(&acc_empty[b], ((j - 2) >> 1) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t kbase = smem_u32(smem + L::kKOff + s * L::kHalves * L::kKBox);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (uint32_t)((kk & 3) * 32);
          const uint64_t ad = umma_desc_k_sw128(qbase + (kk >> 2) * L::kQBox + off);
          const uint64_t bd = umma_desc_k_sw128(kbase + (kk >> 2) * L::kKBox + off);
          umma_bf16(tmem + b * kTcKeys1, ad, bd, idesc, kk > 0);
        }
        umma_commit(&k_empty[s]);
        umma_commit(&acc_full[b]);
        // the stage of tile j - 1 takes tile j - 1 + KS once its MMAs are done
        // (MMA j is queued behind them meanwhile)
        if (j >= 1 && issued < nk) {
          if (!mbar_wait_bounded(&k_empty[(j - 1) % KS], ((j - 1) / KS) & 1)) {
            ok = false;
            break;
          }
          load_k(issued++);
        }
      }
      // unwind: copies still in flight, then every MMA issued
      if (!q_ok) mbar_wait_bounded(q_full, 0);
      for (int t = consumed; t < issued; ++t) mbar_wait_bounded(&k_full[t % KS], (t / KS) & 1);
      umma_commit(mma_done);
      mbar_wait_bounded(mma_done, 0);
    }
    __syncwarp();
  } else {
    // epilogue: thread = query row (tensor-memory lane) x 64 keys of each tile
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    const float sc = a.scale2;
    for (int j = 0; j < nk; ++j) {
      const int b = j & 1;
      if (!mbar_wait_bounded(&acc_full[b], (j >> 1) & 1)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const int kvalid = a.n_ctx - j * kTcKeys1;  // keys of this tile inside the unit
      // this warp's 64 keys (columns 64 grp ..) in one load, one wait, one
      // running-max update and one pass of exponentials
      const int nv = kvalid - grp * 64;
      if (nv > 0) {
        uint32_t r[64];
        tmem_ld64(tmem + lane_base + b * kTcKeys1 + grp * 64, r);
        tmem_ld_wait();
        if (nv < 64) {  // the unit's last keys: the rest belongs to the next unit
#pragma unroll
          for (int i = 0; i < 64; ++i)
            if (i >= nv) r[i] = __float_as_uint(-INFINITY);
        }
        float m4[4] = {__uint_as_float(r[0]), __uint_as_float(r[1]), __uint_as_float(r[2]),
                       __uint_as_float(r[3])};
#pragma unroll
        for (int i = 4; i < 64; i += 8) {
          m4[0] = fmax3(m4[0], __uint_as_float(r[i]), __uint_as_float(r[i + 1]));
          m4[1] = fmax3(m4[1], __uint_as_float(r[i + 2]), __uint_as_float(r[i + 3]));
          m4[2] = fmax3(m4[2], __uint_as_float(r[i + 4]), __uint_as_float(r[i + 5]));
          m4[3] = fmax3(m4[3], __uint_as_float(r[i + 6]), __uint_as_float(r[i + 7]));
        }
        const float cm = fmaxf(fmax3(m4[0], m4[1], m4[2]), m4[3]);
        if (cm > m) {
          ssum *= exp2f((m - cm) * sc);
          m = cm;
        }
        // 2^(x sc - m sc), two lanes of f32x2 arithmetic per instruction
        const float2 sc2 = make_float2(sc, sc), nmc = make_float2(-m * sc, -m * sc);
        float2 s2a = make_float2(0.f, 0.f), s2b = make_float2(0.f, 0.f);
#pragma unroll
        for (int i = 0; i < 64; i += 4) {
          const float2 ea = __ffma2_rn(make_float2(__uint_as_float(r[i]), __uint_as_float(r[i + 1])),
                                       sc2, nmc);
          const float2 eb = __ffma2_rn(
              make_float2(__uint_as_float(r[i + 2]), __uint_as_float(r[i + 3])), sc2, nmc);
          s2a = __fadd2_rn(s2a, make_float2(exp2f(ea.x), exp2f(ea.y)));
          s2b = __fadd2_rn(s2b, make_float2(exp2f(eb.x), exp2f(eb.y)));
        }
        ssum += (s2a.x + s2a.y) + (s2b.x + s2b.y);
      }
      tc_fence_before();
      mbar_arrive(&acc_empty[b]);
    }
  }
  // the four parts of each row meet in shared memory
  float* part = reinterpret_cast<float*>(smem + L::kPartOff);
  if (warp < kTcIssueWarp) {
    part[(grp * 128 + row) * 2] = m;
    part[(grp * 128 + row) * 2 + 1] = ssum;
  }
  __syncthreads();
  if (warp < kTcIssueWarp && grp == 0) {
    float M = -INFINITY;
#pragma unroll
    for (int q = 0; q < kTcGroups; ++q) M = fmaxf(M, part[(q * 128 + row) * 2]);
    float tot = 0.f;
#pragma unroll
    for (int q = 0; q < kTcGroups; ++q)
      tot += part[(q * 128 + row) * 2 + 1] * exp2f((part[(q * 128 + row) * 2] - M) * a.scale2);
    const int r = mt * kTcRows1 + row;
    if (ok && r < a.n_obs) a.lse2[(size_t)unit * a.n_obs + r] = M * a.scale2 + log2f(tot);
  }
  if (!ok) raise_status(a.dev_status, EBD_DEV_TIMEOUT);
  tc_fence_before();
  __syncthreads();
  if (warp == kTcIssueWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

template <int D>
__global__ void __launch_bounds__(kTcThreads, 1)
    score_col_tc_kernel(const __grid_constant__ CUtensorMap tmQ,
                        const __grid_constant__ CUtensorMap tmK, TcArgs a) {
  using L = Tc2Layout<D>;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = align1024(smem_raw);
  float* lse_s = reinterpret_cast<float*>(smem + L::kLseOff);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::kBarOff);
  uint64_t* q_full = bars;
  uint64_t* k_full = bars + 1;     // [2] key stages
  uint64_t* k_empty = bars + 3;    // [2]
  uint64_t* acc_full = bars + 5;   // [2] accumulator halves
  uint64_t* acc_empty = bars + 7;  // [2]
  uint64_t* lse_ready = bars + 9;   // the epilogue staged a unit's row log-sum-exps
  uint64_t* part_ready = bars + 10;  // [2] warps 4-15 left their partial key sums (item parity)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 12);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nkt = (a.n_ctx + kTcKeys2 - 1) / kTcKeys2;
  const int i0 = (int)((long long)blockIdx.x * a.items / gridDim.x);
  const int i1 = (int)((long long)(blockIdx.x + 1) * a.items / gridDim.x);
  const int n = i1 - i0;
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
      mbar_init(&acc_full[s], 1);
      mbar_init(&acc_empty[s], kTcEpi);
    }
    mbar_init(lse_ready, kTcEpi);
    mbar_init(&part_ready[0], kTcEpi - 128);
    mbar_init(&part_ready[1], kTcEpi - 128);
    fence_barrier_init();
  }
  if (warp == kTcIssueWarp) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  bool ok = true;
  const int nq_loads = (a.rows_pad + 255) / 256;  // 256-row TMA boxes of Q

  if (warp == kTcIssueWarp) {
    if (lane == 0 && n > 0) {
      auto load_k = [&](int i) {
        const int item = i0 + i, u = item / nkt, kt = item - u * nkt;
        const int s = i & 1;
        mbar_arrive_expect_tx(&k_full[s], L::kHalves * L::kKBox);
#pragma unroll
        for (int h = 0; h < L::kHalves; ++h)
          tma_load_2d(smem + L::kKOff + (s * L::kHalves + h) * L::kKBox, &tmK, h * 64,
                      u * a.n_ctx + kt * kTcKeys2, &k_full[s]);
      };
      const uint32_t idesc_a = umma_idesc_bf16_f32(128, a.n_a);
      const uint32_t idesc_b = umma_idesc_bf16_f32(128, a.n_b > 0 ? a.n_b : 16);
      const uint32_t qbase = smem_u32(smem);
      int cur_u = -1, qloads = 0;
      bool qwait = false;
      load_k(0);
      for (int i = 0; ok && i < n; ++i) {
        const int item = i0 + i, u = item / nkt;
        const int s = i & 1;
        if (u != cur_u) {  // new unit: Q once every MMA reading the old one is done
          if (i > 0 && !mbar_wait_bounded(&k_empty[s ^ 1], ((i - 1) >> 1) & 1)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(q_full, L::kHalves * nq_loads * 256 * 128);
#pragma unroll
          for (int h = 0; h < L::kHalves; ++h)
            for (int l = 0; l < nq_loads; ++l)
              tma_load_2d(smem + h * L::kQBox + l * 256 * 128, &tmQ, h * 64,
                          u * a.n_obs + l * 256, q_full);
          cur_u = u;
          qwait = true;
        }
        if (i + 1 < n) {
          if (i >= 1 && !mbar_wait_bounded(&k_empty[s ^ 1], ((i - 1) >> 1) & 1)) {
            ok = false;
            break;
          }
          load_k(i + 1);
        }
        if (!mbar_wait_bounded(&k_full[s], (i >> 1) & 1)) {
          ok = false;
          break;
        }
        if (qwait) {
          if (!mbar_wait_bounded(q_full, qloads & 1)) {
            ok = false;
            break;
          }
          ++qloads;
          qwait = false;
        }
        const uint32_t kbase = smem_u32(smem + L::kKOff + s * L::kHalves * L::kKBox);
        for (int hh = 0; hh < 2; ++hh) {
          const int ncols = hh == 0 ? a.n_a : a.n_b;
          if (ncols == 0) continue;
          if (i >= 1 && !mbar_wait_bounded(&acc_empty[hh], (i - 1) & 1)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t row_off = (uint32_t)(hh * a.n_a) * 128u;  // first query row of the half
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t off = (uint32_t)((kk & 3) * 32);
            const uint64_t ad = umma_desc_k_sw128(kbase + (kk >> 2) * L::kKBox + off);
            const uint64_t bd = umma_desc_k_sw128(qbase + (kk >> 2) * L::kQBox + row_off + off);
            umma_bf16(tmem + hh * 256, ad, bd, hh == 0 ? idesc_a : idesc_b, kk > 0);
          }
          umma_commit(&acc_full[hh]);
        }
        if (!ok) break;
        umma_commit(&k_empty[s]);
      }
    }
    __syncwarp();
  } else {
    // epilogue: thread = key (tensor-memory lane); the 32-column chunks of the
    // [A | B] accumulator columns go round-robin to warps w, w + 4, w + 8, w + 12
    const int quarter = warp & 3, grp = warp >> 2;
    const int row = quarter * 32 + lane;
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    float* part = reinterpret_cast<float*>(smem + L::kPartOff);
    const int nch = a.rows_pad / 32;
    int cur_u = -1, par = 0, changes = 0;
    for (int i = 0; i < n; ++i) {
      const int item = i0 + i, u = item / nkt, kt = item - u * nkt;
      if (u != cur_u) {  // this unit's row log-sum-exps (padding rows contribute 0)
        par ^= 1;
        float* ls = lse_s + par * kTcMaxRows;
        for (int r = threadIdx.x; r < a.rows_pad; r += kTcEpi)
          ls[r] = r < a.n_obs ? -a.lse2[(size_t)u * a.n_obs + r] : -INFINITY;
        mbar_arrive(lse_ready);  // release: the rows this thread staged
        if (!mbar_wait_bounded(lse_ready, changes & 1)) {
          ok = false;
          break;
        }
        ++changes;
        cur_u = u;
      }
      const float* ls = lse_s + par * kTcMaxRows;  // minus the row log-sum-exps
      const float2 sc2 = make_float2(a.scale2, a.scale2);
      float2 s2a = make_float2(0.f, 0.f), s2b = make_float2(0.f, 0.f);
      for (int hh = 0; hh < 2; ++hh) {
        const int ncols = hh == 0 ? a.n_a : a.n_b;
        if (ncols == 0) continue;
        if (!mbar_wait_bounded(&acc_full[hh], i & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const int c0 = hh == 0 ? 0 : a.n_a / 32, c1 = hh == 0 ? a.n_a / 32 : nch;
        // first chunk c >= c0 with c % groups == grp
        const int cfirst = c0 + ((grp - c0 % kTcGroups) + kTcGroups) % kTcGroups;
#pragma unroll 1
        for (int c = cfirst; c < c1; c += kTcGroups) {
          uint32_t r[32];
          tmem_ld32(tmem + lane_base + hh * 256 + (c - c0) * 32, r);
          tmem_ld_wait();
          const float4* l4 = reinterpret_cast<const float4*>(ls + c * 32);
#pragma unroll
          for (int t = 0; t < 8; ++t) {
            const float4 lv = l4[t];
            const float2 ea = __ffma2_rn(make_float2(__uint_as_float(r[4 * t]),
                                                     __uint_as_float(r[4 * t + 1])),
                                         sc2, make_float2(lv.x, lv.y));
            const float2 eb = __ffma2_rn(make_float2(__uint_as_float(r[4 * t + 2]),
                                                     __uint_as_float(r[4 * t + 3])),
                                         sc2, make_float2(lv.z, lv.w));
            s2a = __fadd2_rn(s2a, make_float2(exp2f(ea.x), exp2f(ea.y)));
            s2b = __fadd2_rn(s2b, make_float2(exp2f(eb.x), exp2f(eb.y)));
          }
        }
        tc_fence_before();
        mbar_arrive(&acc_empty[hh]);
      }
      if (!ok) break;
      const float sum = (s2a.x + s2a.y) + (s2b.x + s2b.y);
      float* pb = part + (i & 1) * kTcGroups * 128;
      if (grp != 0) {
        pb[grp * 128 + row] = sum;
        mbar_arrive(&part_ready[i & 1]);  // release
      } else {
        // one barrier per buffer: an arrival for item i + 1 can never count
        // toward item i's phase
        if (!mbar_wait_bounded(&part_ready[i & 1], (i >> 1) & 1)) {
          ok = false;
          break;
        }
        float tot = sum;
#pragma unroll
        for (int q = 1; q < kTcGroups; ++q) tot += pb[q * 128 + row];
        const int key = kt * kTcKeys2 + row;
        if (key < a.n_ctx) a.scores[(size_t)u * a.n_ctx + key] = tot;
      }
    }
  }
  if (!ok) raise_status(a.dev_status, EBD_DEV_TIMEOUT);
  tc_fence_before();
  __syncthreads();
  if (warp == kTcIssueWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
static PFN_cuTensorMapEncodeTiled_v12000 tc_encoder() {
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

// [rows, D] bf16 as 2D; box = 64 columns x box_rows rows, 128-byte swizzle.
static bool encode_bf16_rows(CUtensorMap* map, const void* base, long long rows, int D,
                             int box_rows) {
  auto enc = tc_encoder();
  if (!enc) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)D * 2};
  const cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool score_tc_supported(ebd_dtype dtype, int head_dim, int n_obs, const void* q_obs,
                        const void* K) {
  return dtype == EBD_BF16 && (head_dim == 64 || head_dim == 128) && n_obs >= 1 &&
         n_obs <= kTcMaxRows && ((uintptr_t)q_obs & 15u) == 0 && ((uintptr_t)K & 15u) == 0 &&
         tc_encoder() != nullptr;
}

template <int D>
static ebd_status launch_score_tc_t(int units, int n_ctx, int n_obs, const void* q_obs,
                                    const void* K, float* scores, float* lse2,
                                    int32_t* dev_status, cudaStream_t s) {
  CUtensorMap tmQ1, tmK1, tmQ2, tmK2;
  const long long qrows = (long long)units * n_obs, krows = (long long)units * n_ctx;
  if (!encode_bf16_rows(&tmQ1, q_obs, qrows, D, kTcRows1) ||
      !encode_bf16_rows(&tmK1, K, krows, D, kTcKeys1) ||
      !encode_bf16_rows(&tmQ2, q_obs, qrows, D, 256) ||
      !encode_bf16_rows(&tmK2, K, krows, D, kTcKeys2))
    return EBD_ERR_CUDA;
  TcArgs a;
  a.units = units;
  a.n_ctx = n_ctx;
  a.n_obs = n_obs;
  a.mtiles = (n_obs + kTcRows1 - 1) / kTcRows1;
  a.rows_pad = (n_obs + 31) / 32 * 32;
  a.n_a = a.rows_pad < 256 ? a.rows_pad : 256;
  a.n_b = a.rows_pad - a.n_a;
  a.items = units * ((n_ctx + kTcKeys2 - 1) / kTcKeys2);
  a.scale2 = kLog2e / sqrtf((float)D);
  a.lse2 = lse2;
  a.scores = scores;
  a.dev_status = dev_status;
  const int smem1 = Tc1Layout<D>::kBytes, smem2 = Tc2Layout<D>::kBytes;
  if (cudaFuncSetAttribute(score_lse_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           smem1) != cudaSuccess ||
      cudaFuncSetAttribute(score_col_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           smem2) != cudaSuccess)
    return EBD_ERR_CUDA;
  score_lse_tc_kernel<D><<<units * a.mtiles, kTcThreads, smem1, s>>>(tmQ1, tmK1, a);
  ebd_status st = launch_status();
  if (st != EBD_OK) return st;
  const int ctas = a.items < sm_count() ? a.items : sm_count();
  score_col_tc_kernel<D><<<ctas, kTcThreads, smem2, s>>>(tmQ2, tmK2, a);
  return launch_status();
}

ebd_status launch_score_tc(int units, int head_dim, int n_ctx, int n_obs, const void* q_obs,
                           const void* K, float* scores, float* lse, int32_t* dev_status,
                           cudaStream_t s) {
  if ((long long)units * n_ctx >= 0x7fffffffLL || (long long)units * n_obs >= 0x7fffffffLL)
    return EBD_ERR_UNSUPPORTED;
  if (head_dim == 128)
    return launch_score_tc_t<128>(units, n_ctx, n_obs, q_obs, K, scores, lse, dev_status, s);
  if (head_dim == 64)
    return launch_score_tc_t<64>(units, n_ctx, n_obs, q_obs, K, scores, lse, dev_status, s);
  return EBD_ERR_UNSUPPORTED;
}

}  // namespace ebd
