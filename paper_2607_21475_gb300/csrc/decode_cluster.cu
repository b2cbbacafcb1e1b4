// Certified decode on thread-block clusters: one cluster of C = 1, 2, 4 or 8
// CTAs per (batch row, KV head) unit, C the largest that keeps units * C <=
// SMs and gives every CTA at least 8 tiles at capacity (C = 1: one CTA holds
// the whole unit and combines it alone; with more units than SMs those CTAs
// run in waves).
//
// CTA r of a unit's cluster takes tiles [r T / C, (r + 1) T / C) of the unit's
// T active 16-token tiles and splits them into eight contiguous ranges, one
// per warp; every warp streams its range through a private cp.async ring and
// folds it with the same per-tile step as the split-K kernel (decode_tile.cuh).
// The partial states then meet without leaving the chip: the eight warps' in
// shared memory (over the ring), where warp g combines query head g; the
// cluster's CTAs' in the shared memory of CTA 0, written through distributed
// shared memory; after one cluster barrier (which the other CTAs arrive at
// and leave) CTA 0 combines them and writes y_hat, log N_hat, V_hat, b_t and
// r_t (Eq. 3, Theorem 2, Eq. 4).  With one CTA per unit its own combine is
// the head's state and it writes at once.  One launch, no workspace, no merge
// kernel.  Combination rule: w-terms (l, o, cmax, umax) scale by
// e^(M_part - M), u-terms (U, A2, A1) by its square; every part takes A2
// about the unit's centring row (decode.cuh).  Launched as a programmatic
// dependent, each CTA asks L2 for the first tiles of its warps' ranges before
// its dependency wait, so that a layer's stream starts under the tail of the
// launch before it.
#include <cuda_runtime.h>
#include <math.h>

#include "common.cuh"
#include "decode.cuh"
#include "decode_tile.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace ebd {

struct ClusterArgs {
  const __nv_bfloat16* Q;   // [units * G, D]
  const __nv_bfloat16* Kc;  // [units, cap, D]
  const __nv_bfloat16* Vc;
  const float* logw;        // [units, cap]
  const int32_t* n_kept;    // [units]
  int cap;
  int group;                // query heads of this slice (decode.cuh)
  int gstride;              // query heads per unit in the Q / output layout
  int csize;                // CTAs per cluster (per unit)
  int lw_off;               // shared-memory layout, bytes: log(1/pi) stages
  int lead_off;             // CTA records gathered in CTA 0: [csize][G][rec_floats(D)]
  int cen_off;              // the unit's centring row (D bf16), staged for the finish
  float* y;
  float* lse;
  float* var;
  float* b_t;
  float* radius;
  float log_inv_delta;
  float eps0;
  bool exact;               // b_t / radius come from the exact range pass
};

// Combine n <= NMAX records (stride rec_floats(D) floats) of one query head;
// lane holds columns PER * lane .. + PER - 1 of o and A1.
template <int D>
struct HeadSum {
  static constexpr int PER = D / 32;
  float M, l, U, A2, cm, um;
  float o[PER], a1[PER];
  template <int NMAX>
  __device__ __forceinline__ void combine(const float* recs, int n, size_t stride, int lane) {
    M = -INFINITY;
#pragma unroll
    for (int k = 0; k < NMAX; ++k)
      if (k < n) M = fmaxf(M, recs[k * stride + kRecM]);
    l = U = A2 = cm = um = 0.f;
#pragma unroll
    for (int e = 0; e < PER; ++e) o[e] = a1[e] = 0.f;
#pragma unroll
    for (int k = 0; k < NMAX; ++k) {
      if (k >= n) break;
      const float* R = recs + k * stride;
      const float Mk = R[kRecM];
      if (Mk == -INFINITY) continue;
      const float f = expf(Mk - M), f2 = f * f;
      l = fmaf(f, R[kRecL], l);
      U = fmaf(f2, R[kRecU], U);
      A2 = fmaf(f2, R[kRecA2], A2);
      cm = fmaxf(cm, f * R[kRecCmax]);
      um = fmaxf(um, f * R[kRecUmax]);
#pragma unroll
      for (int e = 0; e < PER; ++e) {
        o[e] = fmaf(f, R[kRecHead + PER * lane + e], o[e]);
        a1[e] = fmaf(f2, R[kRecHead + D + PER * lane + e], a1[e]);
      }
    }
  }
};

// L2 prefetch of the first kPrefetchTiles tiles of a warp's range (K, V and
// log(1/pi) rows; the ranges as in the kernel below), its n_kept value read
// now; warp 0 also asks for the unit's query rows (G rows of D bf16 at q_rows)
// and its centring row.  A few tiles per warp keep the prefetched bytes of all
// resident CTAs far below the L2's size (152 x 8 x 32 KB).  The log(1/pi)
// range is trimmed to whole 16-byte blocks.
constexpr int kPrefetchTiles = 4;
template <int D>
__device__ __forceinline__ void prefetch_first_tiles(const __nv_bfloat16* Kc,
                                                     const __nv_bfloat16* Vc, const float* logw,
                                                     const __nv_bfloat16* q_rows, int G,
                                                     const int32_t* n_kept_u, size_t row_base,
                                                     int cap, uint32_t rank, int C, int warp,
                                                     int lane) {
  if (lane > 4) return;
  const int n = min(max(ld_cg_s32(n_kept_u), 0), cap);
  if (warp == 0 && lane >= 3) {
    if (lane == 3) bulk_prefetch_l2(q_rows, (uint32_t)G * D * 2);
    else if (n > 0) bulk_prefetch_l2(Vc + (row_base + centre_row(n)) * D, D * 2);
    return;
  }
  if (lane > 2) return;
  const int T = (n + kMmaTile - 1) / kMmaTile;
  const int c0 = (int)((long long)rank * T / C), c1 = (int)((long long)(rank + 1) * T / C);
  const int tb = c0 + (int)((long long)warp * (c1 - c0) / kMmaConsumers);
  const int te = c0 + (int)((long long)(warp + 1) * (c1 - c0) / kMmaConsumers);
  const int r0 = tb * kMmaTile, r1 = min(min(te, tb + kPrefetchTiles) * kMmaTile, n);
  if (r1 <= r0) return;
  if (lane < 2) {
    const __nv_bfloat16* src = (lane == 0 ? Kc : Vc) + (row_base + r0) * D;
    bulk_prefetch_l2(src, (uint32_t)(r1 - r0) * D * 2);
  } else {
    const uintptr_t b = (reinterpret_cast<uintptr_t>(logw + row_base + r0) + 15) & ~uintptr_t(15);
    const uintptr_t e = reinterpret_cast<uintptr_t>(logw + row_base + r1) & ~uintptr_t(15);
    if (e > b) bulk_prefetch_l2(reinterpret_cast<const void*>(b), (uint32_t)(e - b));
  }
}

template <int D, int S, bool PACK>
__global__ void __launch_bounds__(kMmaThreads, 1) decode_cluster_kernel(ClusterArgs a) {
  using L = MmaTileLayout<D>;
  constexpr int REC = rec_floats(D);
  constexpr int PER = D / 32;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem =
      (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);  // swizzle atoms
  float* lw_s = reinterpret_cast<float*>(smem + a.lw_off);
  float* lead = reinterpret_cast<float*>(smem + a.lead_off);
  const __nv_bfloat16* cen_s = reinterpret_cast<const __nv_bfloat16*>(smem + a.cen_off);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int C = a.csize, G = a.group;
  const uint32_t rank = cluster_rank();
  const int unit = blockIdx.x / C;
  const size_t row_base = (size_t)unit * a.cap;
  // launched as a programmatic dependent, this CTA may start while the
  // predecessor runs: every warp asks L2 for the first tiles of its range,
  // the range taken from a possibly stale n_kept (a hint; L2 prefetches never
  // change what a load returns), so that the stream overlaps the
  // predecessor's tail.  Every value it uses is read after the wait; then a
  // following dependent may launch early.
  prefetch_first_tiles<D>(a.Kc, a.Vc, a.logw, a.Q + (size_t)unit * a.gstride * D, G,
                          a.n_kept + unit, row_base, a.cap, rank, C, warp, lane);
  grid_dependency_wait();
  grid_launch_dependents();
  const int n_u = min(max(__ldg(a.n_kept + unit), 0), a.cap);
  const int T = (n_u + kMmaTile - 1) / kMmaTile;
  const int c0 = (int)((long long)rank * T / C), c1 = (int)((long long)(rank + 1) * T / C);
  const int tb = c0 + (int)((long long)warp * (c1 - c0) / kMmaConsumers);
  const int te = c0 + (int)((long long)(warp + 1) * (c1 - c0) / kMmaConsumers);
  const float kscale = kLog2e * rsqrtf((float)D);

  // CTA 0 stages the centring row for the finish with the first copies
  const int cr = centre_row(n_u);
  if (rank == 0 && warp == 0 && cr >= 0 && lane < D / 8)
    cp_async16(smem + a.cen_off + 16 * lane, a.Vc + (row_base + cr) * D + 8 * lane);
  int issued = 0;
  auto issue_next = [&]() {
    const int t = tb + issued;
    if (t < te) {
      const int stage = warp * S + issued % S;
      tile_copy<D>(smem + (size_t)stage * L::kStageBytes, lw_s + stage * kMmaTile, a.Kc, a.Vc,
                   a.logw, row_base + (size_t)t * kMmaTile, lane);
    }
    cp_async_commit();
    ++issued;
  };
  // the first stages of the ring go out before the query and centring loads,
  // whose latency they then hide
#pragma unroll
  for (int p = 0; p < S - 1; ++p) issue_next();
  TileAcc<D> st;
  tile_acc_begin<D, PACK>(st, a.Q, a.Vc, unit, G, a.gstride, a.cap, n_u, lane);
  int j = 0;
  for (int t = tb; t < te; ++t, ++j) {
    issue_next();  // tile j + S - 1 into the stage tile j - 1 left
    const int s = warp * S + j % S;
    cp_async_wait<S - 1>();  // this lane's copies of tile j are done
    __syncwarp();            // and every lane's
    tile_consume<D, PACK>(st, smem_u32(smem + (size_t)s * L::kStageBytes), lw_s + s * kMmaTile,
                    min(kMmaTile, n_u - t * kMmaTile), lane, kscale);
  }
  cp_async_wait<0>();
  __syncthreads();  // the ring is free: the warps' records go over it

  float* wrec = reinterpret_cast<float*>(smem);  // [warps][G][REC]
  tile_acc_store<D, PACK>(st, wrec + (size_t)warp * G * REC, G, lane);
  __syncthreads();
  HeadSum<D> h;  // this CTA's part of query head `warp`
  if (warp < G)
    h.combine<kMmaConsumers>(wrec + (size_t)warp * REC, kMmaConsumers, (size_t)G * REC, lane);
  if (C > 1) {
    if (warp < G) {  // sent to CTA 0
      const uint32_t dst = cluster_map(smem_u32(lead + ((size_t)rank * G + warp) * REC), 0);
      if (lane == 0) {
        st_cluster4(dst + 4 * kRecM, h.M, h.l, h.U, h.A2);
        st_cluster4(dst + 4 * kRecCmax, h.cm, h.um, 0.f, 0.f);
      }
      if constexpr (PER == 4) {  // 16-byte stores: lane holds columns 4 lane .. + 3
        st_cluster4(dst + 4 * (kRecHead + 4 * lane), h.o[0], h.o[1], h.o[2], h.o[3]);
        st_cluster4(dst + 4 * (kRecHead + D + 4 * lane), h.a1[0], h.a1[1], h.a1[2], h.a1[3]);
      } else {  // lanes 2k and 2k + 1 hold columns 4k .. 4k + 3: even lanes store both
        const float o2 = __shfl_down_sync(0xffffffffu, h.o[0], 1);
        const float o3 = __shfl_down_sync(0xffffffffu, h.o[1], 1);
        const float b2 = __shfl_down_sync(0xffffffffu, h.a1[0], 1);
        const float b3 = __shfl_down_sync(0xffffffffu, h.a1[1], 1);
        if ((lane & 1) == 0) {
          st_cluster4(dst + 4 * (kRecHead + 2 * lane), h.o[0], h.o[1], o2, o3);
          st_cluster4(dst + 4 * (kRecHead + D + 2 * lane), h.a1[0], h.a1[1], b2, b3);
        }
      }
    }
    // every thread arrives; only CTA 0's head warps wait for the records, the
    // other CTAs leave at once and free their SMs for what follows
    cluster_arrive_release();
    if (rank != 0 || warp >= G) return;
    cluster_wait_acquire();
    h.combine<8>(lead + (size_t)warp * REC, C, (size_t)G * REC, lane);
  } else if (warp >= G) {
    return;  // one CTA per unit: its part is the head's whole state
  }
  const long long hq = (long long)unit * a.gstride + warp;
  if (h.M == -INFINITY) {  // no retained row: y = 0, lse = -inf, zero certificate
#pragma unroll
    for (int e = 0; e < PER; ++e) a.y[hq * D + PER * lane + e] = 0.f;
    if (lane == 0) {
      a.lse[hq] = -INFINITY;
      a.var[hq] = 0.f;
      a.b_t[hq] = 0.f;
      a.radius[hq] = 0.f;
    }
    return;
  }
  float c[PER], yv[PER], ynorm, ycnorm, var;
#pragma unroll
  for (int e = 0; e < PER; ++e) c[e] = cr < 0 ? 0.f : __bfloat162float(cen_s[PER * lane + e]);
  finish_head<PER>(h.o, h.a1, c, h.l, h.U, h.A2, yv, ynorm, ycnorm, var);
#pragma unroll
  for (int e = 0; e < PER; ++e) a.y[hq * D + PER * lane + e] = yv[e];
  if (lane == 0) {
    a.lse[hq] = h.M + logf(h.l);
    a.var[hq] = var;
    if (a.exact) {
      a.b_t[hq] = 0.f;  // filled by the exact range pass
    } else {
      const float bt = (h.cm + ycnorm * h.um) / h.l;
      a.b_t[hq] = bt;
      a.radius[hq] = (sqrtf(2.f * var * a.log_inv_delta) + bt * a.log_inv_delta) / (ynorm + a.eps0);
    }
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
template <int D, int S, bool PACK>
static ebd_status launch_cluster_t(const DecodeArgs& d, const ReduceArgs& r, int units, int C,
                                   cudaStream_t s) {
  using L = MmaTileLayout<D>;
  ClusterArgs a;
  a.Q = reinterpret_cast<const __nv_bfloat16*>(d.Q);
  a.Kc = reinterpret_cast<const __nv_bfloat16*>(d.Kc);
  a.Vc = reinterpret_cast<const __nv_bfloat16*>(d.Vc);
  a.logw = d.logw;
  a.n_kept = d.n_kept;
  a.cap = d.cap;
  a.group = d.group;
  a.gstride = d.gstride;
  a.csize = C;
  a.lw_off = kMmaConsumers * S * L::kStageBytes;
  a.lead_off = (int)align_up((size_t)a.lw_off + (size_t)kMmaConsumers * S * kMmaTile * 4, 16);
  a.cen_off = (int)align_up((size_t)a.lead_off + (size_t)C * d.group * rec_floats(D) * 4, 16);
  a.y = r.y;
  a.lse = r.lse;
  a.var = r.var;
  a.b_t = r.b_t;
  a.radius = r.radius;
  a.log_inv_delta = r.log_inv_delta;
  a.eps0 = r.eps0;
  a.exact = r.exact;
  const size_t smem = (size_t)a.cen_off + (size_t)D * 2 + 1024;
  if (cudaFuncSetAttribute(decode_cluster_kernel<D, S, PACK>,
                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
    return EBD_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(units * C));
  cfg.blockDim = dim3(kMmaThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cuda_status(cudaLaunchKernelEx(&cfg, decode_cluster_kernel<D, S, PACK>, a));
}

// Shared memory of a cluster CTA with S ring stages.
static size_t cluster_smem(int D, int S, int C, int G) {
  const size_t stage = (size_t)2 * (D / 64) * kMmaTile * 128;
  const size_t lw = align_up((size_t)kMmaConsumers * S * stage + kMmaConsumers * S * kMmaTile * 4, 16);
  return align_up(lw + (size_t)C * G * rec_floats(D) * 4, 16) + (size_t)D * 2 + 1024;
}

int cluster_decode_size(int units, int cap) {
  const int sms = sm_count();
  if (units < 1) return 0;
  if (units > sms) {
    // more units than SMs: still one CTA per unit, the later ones starting as
    // the first finish (the block scheduler hands them to the SMs that are
    // done first).  Measured on the 32k dialogue shape against the split-K
    // pair: faster when the waves are at least 80% full (256 units, 84%:
    // 83.3 -> 81.9 us; 288 units, 95%: 90.6 -> 86.2 us), much slower when the
    // last wave is thin (160 units: 62.0 -> 79.5 us), and slower for units of
    // more than 512 tiles (the quantisation of long waves)
    const int tiles = cap / kMmaTile;
    const long long waves = (units + sms - 1) / sms;
    if (5LL * units < 4LL * waves * sms) return 0;
    return tiles >= 8 && tiles <= 512 ? 1 : 0;
  }
  int C = 1;  // one CTA per unit (no partner CTAs) when only one fits per SM
  while (C < 8 && 2 * C * units <= sms) C *= 2;
  // measured: the on-chip combine pays off when every CTA has a few tiles to
  // stream (at least 8 at capacity; fewer CTAs per unit rather than the
  // split-K pair when the largest C leaves less: 4k contexts at 5-10% on 4 or
  // 32 units, 15.5-16.9 -> 10.7-12.3 us) and either the clusters cover most
  // SMs or, with fewer CTAs, each CTA's share stays within what one SM
  // streams quickly (at most 160 tiles: on 4 units the single launch beats the
  // split-K pair by up to 20% there, and loses beyond ~250 tiles); otherwise
  // the split-K kernels over every SM are faster
  while (C > 1 && (cap / kMmaTile) / C < 8) C /= 2;
  const int per_cta = (cap / kMmaTile) / C;
  if (per_cta < 8) return 0;
  if (4 * units * C < 3 * sms && per_cta > 160) return 0;
  return C;
}

ebd_status launch_cluster_decode(int head_dim, const DecodeArgs& d, const ReduceArgs& r,
                                 int units, cudaStream_t s) {
  const int C = cluster_decode_size(units, d.cap);
  if (C == 0) return EBD_ERR_UNSUPPORTED;
  const size_t max_smem = 227 * 1024;
  const bool three = cluster_smem(head_dim, 3, C, d.group) <= max_smem;
  const bool pack = d.group <= 4;
  if (head_dim == 128) {
    if (pack)
      return three ? launch_cluster_t<128, 3, true>(d, r, units, C, s)
                   : launch_cluster_t<128, 2, true>(d, r, units, C, s);
    return three ? launch_cluster_t<128, 3, false>(d, r, units, C, s)
                 : launch_cluster_t<128, 2, false>(d, r, units, C, s);
  }
  if (head_dim == 64) {
    if (pack)
      return three ? launch_cluster_t<64, 3, true>(d, r, units, C, s)
                   : launch_cluster_t<64, 2, true>(d, r, units, C, s);
    return three ? launch_cluster_t<64, 3, false>(d, r, units, C, s)
                 : launch_cluster_t<64, 2, false>(d, r, units, C, s);
  }
  return EBD_ERR_UNSUPPORTED;
}

}  // namespace ebd
