// Tensor-core certified decode (bf16 compact cache, head_dim 64/128, G <= 8).
//
// Same quantities as the CUDA-core path (Eq. 3, Theorem 2, Eq. 4): per query
// head an online softmax over logits q.k/sqrt(d) + log(1/pi) carrying
// l = sum w, o = sum w v, U = sum u, A1 = sum u v, A2 = sum u ||v - c||^2
// (c: the unit's centring row, decode.cuh) and the range-bound maxima, with
// u = (1 - pi) w^2.
//
// Two kernels.  The decode kernel is a persistent grid (one CTA per SM) of 8
// warps.  Every CTA first builds the prefix of active 16-token tiles per unit
// (tiles below min(n_kept, cap)) in shared memory (CTA 0 also stores it for
// the merge); the active tiles of all units are then split into equal
// contiguous ranges, one per warp.  A warp's range crosses at most a few
// units; for each unit it meets it writes one partial record, at index
// (unit + global warp), so records never collide and nothing needs clearing.
// The merge kernel (one CTA per query head, launched as a programmatic
// dependent of the decode so its launch overlaps the decode's tail) spreads
// the head's records over its warps, combines them in shared memory and
// writes y_hat, lse, V_hat, b_t and r_t.  The decode kernel is itself launched
// as a programmatic dependent of whatever precedes it (a previous layer's
// merge, say), waiting before its first memory access.
//
// The per-tile step (Q K^T, weights, [w; u] V on mma.sync with hi/lo weight
// parts, ||v||^2, lazy rescale) lives in decode_tile.cuh.
//
// Each warp streams its own tiles: all 32 lanes issue 16-byte cp.async copies
// of K, V (into the 128-byte-swizzled layout ldmatrix reads) and log(1/pi) for
// tile j + 2 into the warp's private 3-stage ring while tile j is consumed, one
// commit group per tile; a stage is read after the lane's wait on its group and
// a warp barrier, and refilled only after the warp has read it.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "decode.cuh"
#include "decode_tile.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace ebd {

constexpr int kMmaStagesPerWarp = 3;
constexpr int kMmaStages = kMmaConsumers * kMmaStagesPerWarp;
constexpr int kMinTilesPerWarp = 4;
constexpr int kLocalUnits = 4096;  // tile prefix kept in shared memory up to this many units

template <int D>
struct MmaLayout {
  static constexpr int kStageBytes = MmaTileLayout<D>::kStageBytes;
  static constexpr int kLogwOff = kMmaStages * kStageBytes;
  static constexpr int kScanOff = kLogwOff + kMmaStages * kMmaTile * 4;  // [kMmaConsumers] ints
  static constexpr int kPlanOff = kScanOff + 64;                  // [kLocalUnits + 1] ints
  static constexpr int kBytes = kPlanOff + (kLocalUnits + 1) * 4 + 1024;  // + alignment slack
};

struct FastArgs {
  const __nv_bfloat16* Q;    // [units * G, D]
  const __nv_bfloat16* Kc;   // [units, cap, D]
  const __nv_bfloat16* Vc;   // [units, cap, D]
  const float* logw;         // [units, cap]
  const int32_t* n_kept;     // [units]
  int32_t* tile_off;         // [units + 1]: written by CTA 0, or by the prefix kernel
  bool plan_done;            // tile_off already holds the prefix (more than kLocalUnits units)
  float* part;               // records [(units + W) * G, rec_floats(D)]
  int32_t* dev_status;
  int units;
  int cap;
  int group;                 // query heads of this slice (decode.cuh)
  int gstride;               // query heads per unit in the Q layout
};

struct MergeArgs {
  const int32_t* tile_off;   // [units + 1]
  const float* part;         // records of the decode kernel
  const __nv_bfloat16* Vc;   // [units, cap, D]: the centring rows
  const int32_t* n_kept;     // [units]
  int cap;
  long long warps;           // warps of the decode grid
  int units;
  int group;                 // query heads of this slice
  int gstride;               // query heads per unit in the output layout
  float* y;                  // [units * G, D]
  float* lse;                // [units * G]
  float* var;
  float* b_t;
  float* radius;
  float log_inv_delta;
  float eps0;
  bool exact;                // b_t / radius come from the exact range pass
};

// Working warps of a decode over Ta active tiles (each gets >= kMinTilesPerWarp).
__host__ __device__ __forceinline__ long long decode_working_warps(long long Ta, long long Wall) {
  const long long Wcap = Ta / kMinTilesPerWarp > 0 ? Ta / kMinTilesPerWarp : 1;
  return Wall < Wcap ? Wall : Wcap;
}

// Largest unit u with tile_off[u] <= t (a unit that holds tile t).
__device__ __forceinline__ int unit_of_tile(const int32_t* tile_off, int units, int t) {
  int lo = 0, hi = units - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (tile_off[mid] <= t) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// Next unit after u that holds at least one tile (tile t exists beyond u).
__device__ __forceinline__ int next_unit(const int32_t* tile_off, int u) {
  ++u;
  while (tile_off[u + 1] == tile_off[u]) ++u;
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

// The same prefix built by one CTA of the decode kernel in shared memory:
// every thread carries the running total itself, so only the per-warp sums of
// one block-wide step pass through `scan`.
__device__ void block_tile_prefix(const int32_t* __restrict__ n_kept, int units, int cap,
                                  int32_t* toff, int* scan) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int carry = 0;
  for (int base = 0; base < units; base += kMmaThreads) {
    const int u = base + tid;
    const int v = u < units ? (min(max(__ldg(n_kept + u), 0), cap) + kMmaTile - 1) / kMmaTile : 0;
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int n = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += n;
    }
    if (lane == 31) scan[warp] = incl;
    __syncthreads();
    int before = 0, total = 0;
#pragma unroll
    for (int w = 0; w < kMmaConsumers; ++w) {
      const int x = scan[w];
      before += w < warp ? x : 0;
      total += x;
    }
    if (u < units) toff[u] = carry + before + incl - v;
    carry += total;
    __syncthreads();  // scan[] is rewritten by the next step
  }
  if (tid == 0) toff[units] = carry;
}

template <int D, bool PACK>
__global__ void __launch_bounds__(kMmaThreads, 1)
    decode_mma_kernel(FastArgs a) {
  using L = MmaLayout<D>;
  constexpr int REC = rec_floats(D);
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem =
      (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);  // swizzle atoms
  float* lw_s = reinterpret_cast<float*>(smem + L::kLogwOff);

  // launched as a programmatic dependent: the previous kernel's outputs
  // (the compact cache, Q) are visible after this wait; nothing is read or
  // written before it
  grid_dependency_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int units = a.units;
  const int32_t* toff = a.tile_off;
  if (!a.plan_done) {
    int32_t* ts = reinterpret_cast<int32_t*>(smem + L::kPlanOff);
    block_tile_prefix(a.n_kept, units, a.cap, ts, reinterpret_cast<int*>(smem + L::kScanOff));
    __syncthreads();
    if (blockIdx.x == 0)
      for (int i = threadIdx.x; i <= units; i += kMmaThreads) a.tile_off[i] = ts[i];
    toff = ts;
  }
  __syncthreads();
  grid_launch_dependents();

  const int Ta = toff[units];
  if (Ta == 0) return;
  const long long W = decode_working_warps(Ta, (long long)gridDim.x * kMmaConsumers);
  // global warp index, consecutive indices on different SMs
  const long long gw = (long long)warp * gridDim.x + blockIdx.x;
  if (gw >= W) return;
  const int tb = (int)(gw * Ta / W);
  const int te = (int)((gw + 1) * Ta / W);
  const int G = a.group;
  const float kscale = kLog2e * rsqrtf((float)D);

  // copies: the warp walks its tiles with one cursor, one commit group per
  // tile (empty past the range)
  int pf_t = tb, pf_u = unit_of_tile(toff, units, tb);
  int pf_lo = toff[pf_u], pf_hi = toff[pf_u + 1];
  int issued = 0;
  auto issue_next = [&]() {
    if (pf_t < te) {
      const int stage = warp * kMmaStagesPerWarp + issued % kMmaStagesPerWarp;
      const size_t row0 = (size_t)pf_u * a.cap + (size_t)(pf_t - pf_lo) * kMmaTile;
      tile_copy<D>(smem + (size_t)stage * L::kStageBytes, lw_s + stage * kMmaTile, a.Kc, a.Vc,
                   a.logw, row0, lane);
      ++pf_t;
      if (pf_t < te && pf_t == pf_hi) {
        pf_u = next_unit(toff, pf_u);
        pf_lo = pf_hi;
        pf_hi = toff[pf_u + 1];
      }
    }
    cp_async_commit();
    ++issued;
  };

  TileAcc<D> st;
  int u = pf_u;
  int seg_end = 0, n_u = 0, seg_start = 0;
  auto begin_segment = [&]() {
    seg_start = toff[u];
    seg_end = toff[u + 1];
    n_u = min(__ldg(a.n_kept + u), a.cap);
    tile_acc_begin<D, PACK>(st, a.Q, a.Vc, u, G, a.gstride, a.cap, n_u, lane);
  };
  auto flush_segment = [&]() {
    tile_acc_store<D, PACK>(st, a.part + (size_t)(u + gw) * G * REC, G, lane);
  };

  // prologue: the first stages of the ring
#pragma unroll
  for (int p = 0; p < kMmaStagesPerWarp - 1; ++p) issue_next();

  begin_segment();
  int j = 0;
  for (int t = tb; t < te; ++t, ++j) {
    issue_next();  // tile j + 2 into the stage tile j - 1 left
    if (t == seg_end) {
      flush_segment();
      u = next_unit(toff, u);
      begin_segment();
    }
    const int n_valid = min(kMmaTile, n_u - (t - seg_start) * kMmaTile);
    const int s = warp * kMmaStagesPerWarp + j % kMmaStagesPerWarp;
    cp_async_wait<kMmaStagesPerWarp - 1>();  // this lane's copies of tile j are done
    __syncwarp();                             // and every lane's
    tile_consume<D, PACK>(st, smem_u32(smem + (size_t)s * L::kStageBytes), lw_s + s * kMmaTile,
                    n_valid, lane, kscale);
  }
  flush_segment();
  cp_async_wait<0>();
}

// Merge the partial records of one query head (Eq. 3, Theorem 2, Eq. 4).  One
// CTA of MW warps per query head.  Warp w takes records w, w + MW, ... four at
// a time (all their loads in flight), keeping a running merge relative to its
// own maximum: every lane reads the same record headers and D/32 columns of o
// and A1.  The MW warp partials are then combined in shared memory by warp 0,
// which writes the outputs.  Records of unit u: index u + gw for every working
// decode warp gw whose tile range meets u.  With CL > 1 a cluster of CL CTAs
// takes one query head, CTA r the r-th of CL equal slices of its records;
// each CTA's combined part goes to CTA 0 through distributed shared memory,
// every thread arrives at the cluster barrier, and CTA 0 (warp 0) waits,
// combines the CL parts in rank order and writes the outputs.
template <int D, int MW, int CL>
__global__ void __launch_bounds__(MW * 32) decode_merge_kernel(MergeArgs a) {
  constexpr int REC = rec_floats(D);
  constexpr int PER = D / 32;
  constexpr int BATCH = 4;
  __shared__ float sh_s[MW][8];  // M, l, U, A2, cmax, umax per warp
  __shared__ __align__(16) float sh_o[MW][D];
  __shared__ __align__(16) float sh_a[MW][D];
  __shared__ __align__(16) float lead[CL][8 + 2 * D];  // CTA parts, in CTA 0
  grid_dependency_wait();
  grid_launch_dependents();  // a following dependent grid may launch now

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = a.group;
  const int head = (int)(blockIdx.x / CL);
  const uint32_t rank = CL > 1 ? cluster_rank() : 0u;
  const int u = head / G, g = head - u * G;
  const long long hq = (long long)u * a.gstride + g;  // output row
  const long long t0 = a.tile_off[u], t1 = a.tile_off[u + 1];
  if (t1 == t0) {  // no retained row: y = 0, lse = -inf, zero certificate
    if (warp == 0 && rank == 0) {
#pragma unroll
      for (int e = 0; e < PER; ++e) a.y[hq * D + PER * lane + e] = 0.f;
      if (lane == 0) {
        a.lse[hq] = -INFINITY;
        a.var[hq] = 0.f;
        a.b_t[hq] = 0.f;
        a.radius[hq] = 0.f;
      }
    }
    return;
  }
  const long long Ta = a.tile_off[a.units];
  const long long W = decode_working_warps(Ta, a.warps);
  const long long gf = ((t0 + 1) * W - 1) / Ta;  // first decode warp meeting u
  const long long gl = (t1 * W - 1) / Ta;        // last
  const int count = (int)(gl - gf + 1);
  // this CTA's slice of the head's records
  const int kb = (int)((long long)rank * count / CL), ke = (int)((long long)(rank + 1) * count / CL);
  const float* R0 = a.part + ((size_t)(u + gf) * G + g) * REC;
  const size_t slot = (size_t)G * REC;

  float Mw = -INFINITY, l = 0.f, U = 0.f, A2 = 0.f, cm = 0.f, um = 0.f;
  float o[PER], a1[PER];
#pragma unroll
  for (int e = 0; e < PER; ++e) o[e] = a1[e] = 0.f;
  for (int k0 = kb + warp; k0 < ke; k0 += BATCH * MW) {
    float4 h[BATCH];
    float2 c[BATCH];
    float ov[BATCH][PER], av[BATCH][PER];
#pragma unroll
    for (int i = 0; i < BATCH; ++i) {
      const int k = k0 + i * MW;
      if (k < ke) {
        const float* R = R0 + k * slot;
        h[i] = __ldcg(reinterpret_cast<const float4*>(R));
        c[i] = __ldcg(reinterpret_cast<const float2*>(R + kRecCmax));
        if constexpr (PER == 4) {
          const float4 x = __ldcg(reinterpret_cast<const float4*>(R + kRecHead) + lane);
          const float4 z = __ldcg(reinterpret_cast<const float4*>(R + kRecHead + D) + lane);
          ov[i][0] = x.x; ov[i][1] = x.y; ov[i][2] = x.z; ov[i][3] = x.w;
          av[i][0] = z.x; av[i][1] = z.y; av[i][2] = z.z; av[i][3] = z.w;
        } else {
          const float2 x = __ldcg(reinterpret_cast<const float2*>(R + kRecHead) + lane);
          const float2 z = __ldcg(reinterpret_cast<const float2*>(R + kRecHead + D) + lane);
          ov[i][0] = x.x; ov[i][1] = x.y;
          av[i][0] = z.x; av[i][1] = z.y;
        }
      } else {
        h[i] = make_float4(-INFINITY, 0.f, 0.f, 0.f);
        c[i] = make_float2(0.f, 0.f);
#pragma unroll
        for (int e = 0; e < PER; ++e) ov[i][e] = av[i][e] = 0.f;
      }
    }
    float mb = Mw;
#pragma unroll
    for (int i = 0; i < BATCH; ++i) mb = fmaxf(mb, h[i].x);
    if (mb > Mw) {  // rescale what this warp holds to the new maximum
      const float s = Mw == -INFINITY ? 0.f : expf(Mw - mb), s2 = s * s;
      l *= s;
      U *= s2;
      A2 *= s2;
      cm *= s;
      um *= s;
#pragma unroll
      for (int e = 0; e < PER; ++e) {
        o[e] *= s;
        a1[e] *= s2;
      }
      Mw = mb;
    }
#pragma unroll
    for (int i = 0; i < BATCH; ++i) {
      if (h[i].x == -INFINITY) continue;
      const float f = expf(h[i].x - Mw), f2 = f * f;
      l = fmaf(f, h[i].y, l);
      U = fmaf(f2, h[i].z, U);
      A2 = fmaf(f2, h[i].w, A2);
      cm = fmaxf(cm, f * c[i].x);
      um = fmaxf(um, f * c[i].y);
#pragma unroll
      for (int e = 0; e < PER; ++e) {
        o[e] = fmaf(f, ov[i][e], o[e]);
        a1[e] = fmaf(f2, av[i][e], a1[e]);
      }
    }
  }
  if (lane == 0) {
    sh_s[warp][0] = Mw;
    sh_s[warp][1] = l;
    sh_s[warp][2] = U;
    sh_s[warp][3] = A2;
    sh_s[warp][4] = cm;
    sh_s[warp][5] = um;
  }
#pragma unroll
  for (int e = 0; e < PER; ++e) {
    sh_o[warp][PER * lane + e] = o[e];
    sh_a[warp][PER * lane + e] = a1[e];
  }
  __syncthreads();

  float Mx = -INFINITY;
  if (warp == 0) {
#pragma unroll
    for (int w = 0; w < MW; ++w) Mx = fmaxf(Mx, sh_s[w][0]);
    l = U = A2 = cm = um = 0.f;
#pragma unroll
    for (int e = 0; e < PER; ++e) o[e] = a1[e] = 0.f;
#pragma unroll
    for (int w = 0; w < MW; ++w) {
      const float Ms = sh_s[w][0];
      if (Ms == -INFINITY) continue;
      const float f = expf(Ms - Mx), f2 = f * f;
      l = fmaf(f, sh_s[w][1], l);
      U = fmaf(f2, sh_s[w][2], U);
      A2 = fmaf(f2, sh_s[w][3], A2);
      cm = fmaxf(cm, f * sh_s[w][4]);
      um = fmaxf(um, f * sh_s[w][5]);
#pragma unroll
      for (int e = 0; e < PER; ++e) {
        o[e] = fmaf(f, sh_o[w][PER * lane + e], o[e]);
        a1[e] = fmaf(f2, sh_a[w][PER * lane + e], a1[e]);
      }
    }
  }
  if constexpr (CL > 1) {
    if (warp == 0) {  // this CTA's part, to CTA 0
      const uint32_t dst = cluster_map(smem_u32(&lead[rank][0]), 0);
      if (lane == 0) {
        st_cluster4(dst, Mx, l, U, A2);
        st_cluster4(dst + 16, cm, um, 0.f, 0.f);
      }
#pragma unroll
      for (int e = 0; e < PER; e += 2) {
        asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" ::"r"(dst + 4 * (8 + PER * lane + e)),
                     "f"(o[e]), "f"(o[e + 1]) : "memory");
        asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" ::"r"(dst + 4 * (8 + D + PER * lane + e)),
                     "f"(a1[e]), "f"(a1[e + 1]) : "memory");
      }
    }
    // every thread arrives; CTA 0's warp 0 alone waits for the parts
    cluster_arrive_release();
    if (rank != 0 || warp != 0) return;
    cluster_wait_acquire();
    Mx = -INFINITY;
#pragma unroll
    for (int r = 0; r < CL; ++r) Mx = fmaxf(Mx, lead[r][0]);
    l = U = A2 = cm = um = 0.f;
#pragma unroll
    for (int e = 0; e < PER; ++e) o[e] = a1[e] = 0.f;
#pragma unroll
    for (int r = 0; r < CL; ++r) {
      const float Ms = lead[r][0];
      if (Ms == -INFINITY) continue;
      const float f = expf(Ms - Mx), f2 = f * f;
      l = fmaf(f, lead[r][1], l);
      U = fmaf(f2, lead[r][2], U);
      A2 = fmaf(f2, lead[r][3], A2);
      cm = fmaxf(cm, f * lead[r][4]);
      um = fmaxf(um, f * lead[r][5]);
#pragma unroll
      for (int e = 0; e < PER; ++e) {
        o[e] = fmaf(f, lead[r][8 + PER * lane + e], o[e]);
        a1[e] = fmaf(f2, lead[r][8 + D + PER * lane + e], a1[e]);
      }
    }
  } else {
    if (warp != 0) return;
  }
  float c[PER], yv[PER], ynorm, ycnorm, var;
  load_centre<__nv_bfloat16, D, PER>(a.Vc, u, a.cap, min(max(__ldg(a.n_kept + u), 0), a.cap),
                                     lane, c);
  finish_head<PER>(o, a1, c, l, U, A2, yv, ynorm, ycnorm, var);
  if constexpr (PER == 4)
    *reinterpret_cast<float4*>(a.y + hq * D + 4 * lane) = make_float4(yv[0], yv[1], yv[2], yv[3]);
  else
    *reinterpret_cast<float2*>(a.y + hq * D + 2 * lane) = make_float2(yv[0], yv[1]);
  if (lane == 0) {
    a.lse[hq] = Mx + logf(l);
    a.var[hq] = var;
    if (a.exact) {
      a.b_t[hq] = 0.f;  // filled by the exact range pass
    } else {
      const float bt = (cm + ycnorm * um) / l;
      a.b_t[hq] = bt;
      a.radius[hq] = (sqrtf(2.f * var * a.log_inv_delta) + bt * a.log_inv_delta) / (ynorm + a.eps0);
    }
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
bool fast_decode_supported(ebd_dtype dtype, int group, int head_dim, int capacity) {
  return dtype == EBD_BF16 && (head_dim == 64 || head_dim == 128) && group >= 1 && group <= 8 &&
         capacity % kMmaTile == 0;
}

// Workspace of the tensor-core path: the tile prefix, then the records.
static size_t fast_plan_bytes(long long units) {
  return align_up((size_t)(units + 1) * sizeof(int32_t), 256);
}

void fast_decode_plan(DecodePlan& p, long long units, int group, int head_dim) {
  p.ctas = sm_count();
  const long long W = (long long)p.ctas * kMmaConsumers;
  p.ws_bytes = fast_plan_bytes(units) +
               align_up((size_t)(units + W) * group * rec_floats(head_dim) * sizeof(float), 256);
}


bool fast_decode_usable(const DecodeArgs& a, const ReduceArgs& r, int units) {
  return aligned16(a.Kc) && aligned16(a.Vc) && aligned16(a.logw) && aligned16(a.Q) &&
         aligned16(r.y) && (long long)units * a.cap < 0x7fffffffLL;
}

template <int D>
static ebd_status launch_fast_t(const DecodePlan& plan, const DecodeArgs& a, const ReduceArgs& r,
                                int units, void* ws, cudaStream_t s) {
  int32_t* tile_off = reinterpret_cast<int32_t*>(ws);
  float* recs = reinterpret_cast<float*>(reinterpret_cast<char*>(ws) + fast_plan_bytes(units));
  const bool plan_done = units > kLocalUnits;
  if (plan_done) {
    decode_tile_plan_kernel<<<1, 1024, 0, s>>>(a.n_kept, units, a.cap, tile_off);
    const ebd_status st = launch_status();
    if (st != EBD_OK) return st;
  }
  FastArgs f;
  f.Q = reinterpret_cast<const __nv_bfloat16*>(a.Q);
  f.Kc = reinterpret_cast<const __nv_bfloat16*>(a.Kc);
  f.Vc = reinterpret_cast<const __nv_bfloat16*>(a.Vc);
  f.logw = a.logw;
  f.n_kept = a.n_kept;
  f.tile_off = tile_off;
  f.plan_done = plan_done;
  f.part = recs;
  f.dev_status = a.dev_status;
  f.units = units;
  f.cap = a.cap;
  f.group = a.group;
  f.gstride = a.gstride;
  const int smem = MmaLayout<D>::kBytes;
  const bool pack = a.group <= 4;
  auto kern = pack ? decode_mma_kernel<D, true> : decode_mma_kernel<D, false>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
      cudaSuccess)
    return EBD_ERR_CUDA;
  {
    // programmatic dependent of whatever precedes it in the stream: its launch
    // overlaps that kernel's tail (the kernel waits before touching memory)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)plan.ctas);
    cfg.blockDim = dim3(kMmaThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const ebd_status st = cuda_status(cudaLaunchKernelEx(&cfg, kern, f));
    if (st != EBD_OK) return st;
  }

  MergeArgs m;
  m.tile_off = tile_off;
  m.part = recs;
  m.Vc = f.Vc;
  m.n_kept = a.n_kept;
  m.cap = a.cap;
  m.warps = (long long)plan.ctas * kMmaConsumers;
  m.units = units;
  m.group = a.group;
  m.gstride = a.gstride;
  m.y = r.y;
  m.lse = r.lse;
  m.var = r.var;
  m.b_t = r.b_t;
  m.radius = r.radius;
  m.log_inv_delta = r.log_inv_delta;
  m.eps0 = r.eps0;
  m.exact = r.exact;
  cudaLaunchConfig_t cfg = {};
  const long long heads = (long long)units * a.group;
  cfg.gridDim = dim3((unsigned)heads);
  // a few records per head: 2 warps (one wave of CTAs); many: 8 warps;
  // hundreds (few long units): clusters of 4 CTAs of 16 warps per head, so
  // that more SMs share the records and each warp keeps few rounds of record
  // loads in flight
  const long long per_unit = (long long)plan.ctas * kMmaConsumers / units;
  const int mw = per_unit > 96 ? 16 : per_unit > 12 ? 8 : 2;
  cfg.blockDim = dim3(mw * 32);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (mw == 16) {
    constexpr int CL = 4;
    cfg.gridDim = dim3((unsigned)(heads * CL));
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = CL;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.numAttrs = 2;
    return cuda_status(cudaLaunchKernelEx(&cfg, decode_merge_kernel<D, 16, CL>, m));
  }
  if (mw == 8) return cuda_status(cudaLaunchKernelEx(&cfg, decode_merge_kernel<D, 8, 1>, m));
  return cuda_status(cudaLaunchKernelEx(&cfg, decode_merge_kernel<D, 2, 1>, m));
}

ebd_status launch_fast_decode(ebd_dtype dtype, int head_dim, const DecodePlan& plan,
                              const DecodeArgs& a, const ReduceArgs& r, int units, void* ws,
                              cudaStream_t stream) {
  if (dtype != EBD_BF16) return EBD_ERR_UNSUPPORTED;
  // few units: one cluster of CTAs per unit, combined on chip (decode_cluster.cu);
  // should that launch be refused, the split-K kernels below take the request
  if (cluster_decode_size(units, a.cap) > 0) {
    if (launch_cluster_decode(head_dim, a, r, units, stream) == EBD_OK) return EBD_OK;
    cudaGetLastError();
  }
  if (head_dim == 128) return launch_fast_t<128>(plan, a, r, units, ws, stream);
  if (head_dim == 64) return launch_fast_t<64>(plan, a, r, units, ws, stream);
  return EBD_ERR_UNSUPPORTED;
}

}  // namespace ebd
