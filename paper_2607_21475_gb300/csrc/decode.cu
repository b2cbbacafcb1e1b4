// Certified decode over the compact cache (Section 3.3 Eq. 3, Theorem 2,
// Section 3.4 Eq. 4 of the paper), split-K over the retained tokens.
//
// Each split of each (batch row, KV head) unit streams its K_c, V_c, logw_c
// rows once and keeps, per query head of the group, an online-softmax state
// relative to its running maximum logit M:
//   l  = sum w_i                    w_i = exp(q.k_i/sqrt(d) + log(1/pi_i) - M)
//   o  = sum w_i v_i                (Hajek numerator, Eq. 3)
//   U  = sum u_i,  u_i = (1 - pi_i) w_i^2   (Theorem 2 weights)
//   A1 = sum u_i v_i,  A2 = sum u_i ||v_i - c||^2  (c: the unit's centring row)
//   cmax = max sqrt(u_i) ||v_i - c||,  umax = max sqrt(u_i)   (range-term bound)
// A maximum increase by D rescales the w-terms by e^-D and the u-terms by
// e^-2D.  The reduce kernel merges the splits the same way and finishes
//   y_hat = o / l,   lse = M + log l  (= log N_hat),
//   V_hat = (A2 - 2 (y_hat - c).(A1 - U c) + ||y_hat - c||^2 U) / l^2
//         = sum u_i ||v_i - y_hat||^2 / l^2,
//   b_t   = (cmax + ||y_hat - c|| umax) / l   (bound; >= the definition),
//   r_t   = (sqrt(2 V_hat ln(1/delta)) + b_t ln(1/delta)) / (||y_hat|| + eps0).
// The exact range term, max_i sqrt(u_i) ||v_i - y_hat|| / l, needs y_hat and is
// a second pass over the tail rows (EBD_RANGE_EXACT).
//
// This file holds the CUDA-core path (any supported dtype, head_dim 64/128, at
// most 8 query heads per pass) and the entry point, which decodes a group of
// up to 16 heads in slices.  The record layout and reduce are shared with the
// tensor-core path.
#include <cuda_runtime.h>
#include <math.h>

#include "common.cuh"
#include "decode.cuh"
#include "internal.h"

namespace ebd {

constexpr int kGenThreads = 128;
constexpr int kGenWarps = kGenThreads / 32;

template <typename T, int D, int GM>
__global__ void __launch_bounds__(kGenThreads) decode_generic_kernel(DecodeArgs a) {
  constexpr int E = D / 32;
  constexpr int REC = rec_floats(D);
  __shared__ float st[kGenWarps][GM][REC];
  const int unit = blockIdx.y, split = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = a.group;
  const int n = min(a.n_kept[unit], a.cap);
  const int t0 = split * a.tokens_per_split;
  const int t1 = min(n, t0 + a.tokens_per_split);
  const float scale = rsqrtf((float)D);
  const T* Q = (const T*)a.Q + (size_t)unit * a.gstride * D;
  const T* Kc = (const T*)a.Kc + (size_t)unit * a.cap * D;
  const T* Vc = (const T*)a.Vc + (size_t)unit * a.cap * D;
  const float* lw = a.logw + (size_t)unit * a.cap;
  // the unit's centring row (zeros for an empty unit): A2 is taken about it
  float c[E];
  {
    const int cr = centre_row(max(n, 0));
#pragma unroll
    for (int j = 0; j < E; ++j) c[j] = cr < 0 ? 0.f : to_f32(Vc[(size_t)cr * D + lane + 32 * j]);
  }

  float q[GM][E], o[GM][E], a1[GM][E];
  float M[GM], l[GM], U[GM], A2[GM], cmax[GM], umax[GM];
#pragma unroll
  for (int g = 0; g < GM; ++g) {
#pragma unroll
    for (int j = 0; j < E; ++j) {
      q[g][j] = g < G ? to_f32(Q[(size_t)g * D + lane + 32 * j]) * scale : 0.f;
      o[g][j] = 0.f;
      a1[g][j] = 0.f;
    }
    M[g] = -INFINITY;
    l[g] = U[g] = A2[g] = cmax[g] = umax[g] = 0.f;
  }
  for (int t = t0 + warp; t < t1; t += kGenWarps) {
    float k[E], v[E];
#pragma unroll
    for (int j = 0; j < E; ++j) {
      k[j] = to_f32(Kc[(size_t)t * D + lane + 32 * j]);
      v[j] = to_f32(Vc[(size_t)t * D + lane + 32 * j]);
    }
    const float lwt = lw[t];
    const float omp = -expm1f(-lwt);  // 1 - pi
    const float sq = sqrtf(omp);
    float vc2 = 0.f;
#pragma unroll
    for (int j = 0; j < E; ++j) {
      const float dv = v[j] - c[j];
      vc2 = fmaf(dv, dv, vc2);
    }
    vc2 = warp_sum(vc2);
    const float vn = sqrtf(vc2);  // ||v - c||
#pragma unroll
    for (int g = 0; g < GM; ++g) {
      if (g >= G) break;
      float dot = 0.f;
#pragma unroll
      for (int j = 0; j < E; ++j) dot = fmaf(q[g][j], k[j], dot);
      const float x = warp_sum(dot) + lwt;
      if (x > M[g]) {
        const float f = expf(M[g] - x), f2 = f * f;
        l[g] *= f;
        U[g] *= f2;
        A2[g] *= f2;
        cmax[g] *= f;
        umax[g] *= f;
#pragma unroll
        for (int j = 0; j < E; ++j) {
          o[g][j] *= f;
          a1[g][j] *= f2;
        }
        M[g] = x;
      }
      const float w = expf(x - M[g]);
      const float u = omp * w * w;
      const float su = sq * w;
      l[g] += w;
      U[g] += u;
      A2[g] = fmaf(u, vc2, A2[g]);
      cmax[g] = fmaxf(cmax[g], su * vn);
      umax[g] = fmaxf(umax[g], su);
#pragma unroll
      for (int j = 0; j < E; ++j) {
        o[g][j] = fmaf(w, v[j], o[g][j]);
        a1[g][j] = fmaf(u, v[j], a1[g][j]);
      }
    }
  }
  // merge the warps' states
#pragma unroll
  for (int g = 0; g < GM; ++g) {
    if (lane == 0) {
      st[warp][g][kRecM] = M[g];
      st[warp][g][kRecL] = l[g];
      st[warp][g][kRecU] = U[g];
      st[warp][g][kRecA2] = A2[g];
      st[warp][g][kRecCmax] = cmax[g];
      st[warp][g][kRecUmax] = umax[g];
    }
#pragma unroll
    for (int j = 0; j < E; ++j) {
      st[warp][g][kRecHead + lane + 32 * j] = o[g][j];
      st[warp][g][kRecHead + D + lane + 32 * j] = a1[g][j];
    }
  }
  __syncthreads();
  float* out = a.part + ((size_t)unit * a.splits + split) * (size_t)G * REC;
  for (int idx = threadIdx.x; idx < G * REC; idx += kGenThreads) {
    const int g = idx / REC, e = idx - g * REC;
    float Mx = -INFINITY;
#pragma unroll
    for (int w = 0; w < kGenWarps; ++w) Mx = fmaxf(Mx, st[w][g][kRecM]);
    float r;
    if (e == kRecM) {
      r = Mx;
    } else {
      const bool sq2 = rec_is_squared(e, D);
      const bool is_max = (e == kRecCmax || e == kRecUmax);
      r = 0.f;
#pragma unroll
      for (int w = 0; w < kGenWarps; ++w) {
        const float Mw = st[w][g][kRecM];
        const float f = (Mw == -INFINITY) ? 0.f : expf(Mw - Mx);
        const float x = st[w][g][e] * (sq2 ? f * f : f);
        r = is_max ? fmaxf(r, x) : r + x;
      }
    }
    out[idx] = r;
  }
}

// Merge the partial records of one query head and finish Eq. (3), Theorem 2,
// Eq. (4) (CUDA-core path; the tensor-core kernel merges in place).  One warp
// per query head: lanes take 32 records at a time (scale factors and scalar
// moments), then every lane streams its D/32 columns of each record, records
// u*splits .. u*splits + splits - 1.
constexpr int kReduceWarps = 4;

template <typename T, int D>
__global__ void __launch_bounds__(kReduceWarps * 32) decode_reduce_kernel(ReduceArgs a,
                                                                          int n_heads) {
  constexpr int REC = rec_floats(D);
  constexpr int PER = D / 32;
  const int lane = threadIdx.x & 31;
  const int hs = blockIdx.x * kReduceWarps + (threadIdx.x >> 5);  // head of the slice
  if (hs >= n_heads) return;
  const int G = a.group;
  const int unit = hs / G, g = hs - unit * G;
  const int hq = unit * a.gstride + g;  // output row
  const long long first = (long long)unit * a.splits;
  const int count = a.splits;
  const size_t slot = (size_t)G * REC;
  const float* R0 = a.part + ((size_t)first * G + g) * REC;
  float Mx = -INFINITY;
  for (int s = lane; s < count; s += 32) Mx = fmaxf(Mx, R0[s * slot + kRecM]);
  Mx = warp_max(Mx);
  if (Mx == -INFINITY) {  // empty unit
#pragma unroll
    for (int e = 0; e < PER; ++e) a.y[(size_t)hq * D + PER * lane + e] = 0.f;
    if (lane == 0) {
      a.lse[hq] = -INFINITY;
      a.var[hq] = 0.f;
      a.b_t[hq] = 0.f;
      a.radius[hq] = 0.f;
    }
    return;
  }
  float l = 0.f, U = 0.f, A2 = 0.f, cmax = 0.f, umax = 0.f;
  float o[PER], a1[PER];
#pragma unroll
  for (int e = 0; e < PER; ++e) o[e] = a1[e] = 0.f;
  for (int s0 = 0; s0 < count; s0 += 32) {
    float f = 0.f;
    if (s0 + lane < count) {
      const float* R = R0 + (s0 + lane) * slot;
      const float Ms = R[kRecM];
      if (Ms != -INFINITY) {
        f = expf(Ms - Mx);
        const float f2 = f * f;
        l = fmaf(f, R[kRecL], l);
        U = fmaf(f2, R[kRecU], U);
        A2 = fmaf(f2, R[kRecA2], A2);
        cmax = fmaxf(cmax, f * R[kRecCmax]);
        umax = fmaxf(umax, f * R[kRecUmax]);
      }
    }
    const int nrec = min(32, count - s0);
#pragma unroll 4
    for (int k = 0; k < nrec; ++k) {
      const float fk = __shfl_sync(0xffffffffu, f, k);
      const float f2k = fk * fk;
      const float* Rk = R0 + (s0 + k) * slot + kRecHead + PER * lane;
      if constexpr (PER == 4) {
        const float4 ov = *reinterpret_cast<const float4*>(Rk);
        const float4 av = *reinterpret_cast<const float4*>(Rk + D);
        o[0] = fmaf(fk, ov.x, o[0]);
        o[1] = fmaf(fk, ov.y, o[1]);
        o[2] = fmaf(fk, ov.z, o[2]);
        o[3] = fmaf(fk, ov.w, o[3]);
        a1[0] = fmaf(f2k, av.x, a1[0]);
        a1[1] = fmaf(f2k, av.y, a1[1]);
        a1[2] = fmaf(f2k, av.z, a1[2]);
        a1[3] = fmaf(f2k, av.w, a1[3]);
      } else {
        const float2 ov = *reinterpret_cast<const float2*>(Rk);
        const float2 av = *reinterpret_cast<const float2*>(Rk + D);
        o[0] = fmaf(fk, ov.x, o[0]);
        o[1] = fmaf(fk, ov.y, o[1]);
        a1[0] = fmaf(f2k, av.x, a1[0]);
        a1[1] = fmaf(f2k, av.y, a1[1]);
      }
    }
  }
  l = warp_sum(l);
  U = warp_sum(U);
  A2 = warp_sum(A2);
  cmax = warp_max(cmax);
  umax = warp_max(umax);
  float c[PER], yv[PER], ynorm, ycnorm, var;
  load_centre<T, D, PER>(static_cast<const T*>(a.Vc), unit, a.cap,
                         min(max(a.n_kept[unit], 0), a.cap), lane, c);
  finish_head<PER>(o, a1, c, l, U, A2, yv, ynorm, ycnorm, var);
#pragma unroll
  for (int e = 0; e < PER; ++e) a.y[(size_t)hq * D + PER * lane + e] = yv[e];
  if (lane == 0) {
    a.lse[hq] = Mx + logf(l);
    a.var[hq] = var;
    if (a.exact) {
      a.b_t[hq] = 0.f;  // filled by the exact range pass
    } else {
      const float bt = (cmax + ycnorm * umax) / l;
      a.b_t[hq] = bt;
      a.radius[hq] = (sqrtf(2.f * var * a.log_inv_delta) + bt * a.log_inv_delta) / (ynorm + a.eps0);
    }
  }
}

// EBD_RANGE_EXACT, pass 2: max over tail rows of sqrt(1-pi_i) w_i ||v_i - y_hat|| / N_hat.
template <typename T, int D, int GM>
__global__ void __launch_bounds__(kGenThreads) decode_exact_range_kernel(DecodeArgs a) {
  constexpr int E = D / 32;
  __shared__ float smax[kGenWarps][GM];
  const int unit = blockIdx.y, split = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = a.group;
  const int n = min(a.n_kept[unit], a.cap);
  const int t0 = split * a.tokens_per_split;
  const int t1 = min(n, t0 + a.tokens_per_split);
  const float scale = rsqrtf((float)D);
  const size_t hq0 = (size_t)unit * a.gstride;
  const T* Q = (const T*)a.Q + hq0 * D;
  const T* Kc = (const T*)a.Kc + (size_t)unit * a.cap * D;
  const T* Vc = (const T*)a.Vc + (size_t)unit * a.cap * D;
  const float* lw = a.logw + (size_t)unit * a.cap;
  float q[GM][E], yv[GM][E], lse[GM], best[GM];
#pragma unroll
  for (int g = 0; g < GM; ++g) {
#pragma unroll
    for (int j = 0; j < E; ++j) {
      q[g][j] = g < G ? to_f32(Q[(size_t)g * D + lane + 32 * j]) * scale : 0.f;
      yv[g][j] = g < G ? a.y[(hq0 + g) * D + lane + 32 * j] : 0.f;
    }
    lse[g] = g < G ? a.lse[hq0 + g] : 0.f;
    best[g] = 0.f;
  }
  for (int t = t0 + warp; t < t1; t += kGenWarps) {
    const float lwt = lw[t];
    if (!(lwt > 0.f)) continue;  // pi = 1: not in the tail sample
    float k[E], v[E];
#pragma unroll
    for (int j = 0; j < E; ++j) {
      k[j] = to_f32(Kc[(size_t)t * D + lane + 32 * j]);
      v[j] = to_f32(Vc[(size_t)t * D + lane + 32 * j]);
    }
    const float sq = sqrtf(-expm1f(-lwt));
#pragma unroll
    for (int g = 0; g < GM; ++g) {
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
      const float p = expf(x - lse[g]);  // w_i / N_hat
      best[g] = fmaxf(best[g], sq * p * sqrtf(dist));
    }
  }
  if (lane == 0) {
#pragma unroll
    for (int g = 0; g < GM; ++g) smax[warp][g] = best[g];
  }
  __syncthreads();
  if (threadIdx.x < G) {
    float m = 0.f;
#pragma unroll
    for (int w = 0; w < kGenWarps; ++w) m = fmaxf(m, smax[w][threadIdx.x]);
    // non-negative floats order like their bit patterns
    atomicMax((unsigned int*)&a.b_t[hq0 + threadIdx.x], __float_as_uint(m));
  }
}

template <int D>
__global__ void decode_radius_kernel(ReduceArgs a, int n_heads) {
  const int hq = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (hq >= n_heads) return;
  float yy = 0.f;
  for (int e = lane; e < D; e += 32) {
    const float y = a.y[(size_t)hq * D + e];
    yy = fmaf(y, y, yy);
  }
  yy = warp_sum(yy);
  if (lane == 0) {
    const float bt = a.b_t[hq], var = a.var[hq];
    a.radius[hq] = (sqrtf(2.f * var * a.log_inv_delta) + bt * a.log_inv_delta) / (sqrtf(yy) + a.eps0);
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
template <typename T, int D, int GM>
static ebd_status launch_generic_t(const DecodeArgs& a, int units, cudaStream_t s) {
  dim3 grid(a.splits, units);
  decode_generic_kernel<T, D, GM><<<grid, kGenThreads, 0, s>>>(a);
  return launch_status();
}

template <typename T, int D, int GM>
static ebd_status launch_exact_t(const DecodeArgs& a, int units, cudaStream_t s) {
  dim3 grid(a.splits, units);
  decode_exact_range_kernel<T, D, GM><<<grid, kGenThreads, 0, s>>>(a);
  return launch_status();
}

template <typename T, int D>
static ebd_status dispatch_g(bool exact, const DecodeArgs& a, int units, cudaStream_t s) {
  const int G = a.group;
  if (G <= 1) return exact ? launch_exact_t<T, D, 1>(a, units, s) : launch_generic_t<T, D, 1>(a, units, s);
  if (G <= 2) return exact ? launch_exact_t<T, D, 2>(a, units, s) : launch_generic_t<T, D, 2>(a, units, s);
  if (G <= 4) return exact ? launch_exact_t<T, D, 4>(a, units, s) : launch_generic_t<T, D, 4>(a, units, s);
  return exact ? launch_exact_t<T, D, 8>(a, units, s) : launch_generic_t<T, D, 8>(a, units, s);
}

static ebd_status dispatch_generic(bool exact, ebd_dtype dt, int D, const DecodeArgs& a, int units,
                                   cudaStream_t s) {
  if (dt == EBD_F32) {
    if (D == 64) return dispatch_g<float, 64>(exact, a, units, s);
    if (D == 128) return dispatch_g<float, 128>(exact, a, units, s);
  } else {
    if (D == 64) return dispatch_g<__nv_bfloat16, 64>(exact, a, units, s);
    if (D == 128) return dispatch_g<__nv_bfloat16, 128>(exact, a, units, s);
  }
  return EBD_ERR_UNSUPPORTED;
}

static DecodePlan plan_generic(long long units, int group, int head_dim, int capacity) {
  // CUDA-core path: ~8 resident CTAs per SM, at least 32 tokens per split
  DecodePlan p;
  const long long target = (long long)sm_count() * 8;
  long long splits = (target + units - 1) / units;
  const long long max_splits = (capacity + 31) / 32;
  if (splits > max_splits) splits = max_splits;
  if (splits < 1) splits = 1;
  if (splits > 65535) splits = 65535;
  p.splits = (int)splits;
  p.tokens_per_split = (int)((capacity + splits - 1) / splits);
  p.ws_bytes = align_up((size_t)units * p.splits * group * rec_floats(head_dim) * sizeof(float), 256);
  return p;
}

// Groups of more than kSliceHeads query heads are decoded in slices of at
// most kSliceHeads heads, one pass over the compact cache each (the
// tensor-core tile holds 8 query rows and their 8 u rows).
constexpr int kSliceHeads = 8;
static int decode_slices(int group) { return (group + kSliceHeads - 1) / kSliceHeads; }

DecodePlan plan_decode(ebd_dtype dtype, int batch, int n_kv_heads, int group, int head_dim,
                       int capacity) {
  const long long units = (long long)batch * n_kv_heads;
  const int slices = decode_slices(group);
  group = (group + slices - 1) / slices;  // the largest slice; slices reuse the workspace
  DecodePlan p = plan_generic(units, group, head_dim, capacity);
  if (fast_decode_supported(dtype, group, head_dim, capacity)) {
    const size_t generic_ws = p.ws_bytes;
    p.fast = true;
    fast_decode_plan(p, units, group, head_dim);
    if (p.ws_bytes < generic_ws) p.ws_bytes = generic_ws;  // either path fits
  }
  return p;
}

}  // namespace ebd

using namespace ebd;

extern "C" size_t ebd_decode_workspace_bytes(ebd_dtype dtype, int32_t batch, int32_t n_kv_heads,
                                             int32_t group, int32_t head_dim, int32_t capacity) {
  if (batch < 1 || n_kv_heads < 1 || group < 1 || head_dim < 1 || capacity < 1) return 0;
  return plan_decode(dtype, batch, n_kv_heads, group, head_dim, capacity).ws_bytes;
}

extern "C" size_t ebd_workspace_bytes(const ebd_design* design, int32_t capacity) {
  if (!design || capacity < 1) return 0;
  const ebd_design& d = *design;
  size_t need = ebd_evict_workspace_bytes(design, 0);
  const size_t scored = ebd_evict_workspace_bytes(design, 64 * d.group);
  if (scored > need) need = scored;
  for (ebd_dtype t : {EBD_F32, EBD_BF16}) {
    const size_t dec =
        ebd_decode_workspace_bytes(t, d.batch, d.n_kv_heads, d.group, d.head_dim, capacity);
    if (dec > need) need = dec;
  }
  return need;
}

namespace ebd {

ebd_status check_decode_args(ebd_dtype dtype, int32_t batch, int32_t n_kv_heads, int32_t group,
                             int32_t head_dim, const void* Q, const void* K_c, const void* V_c,
                             const float* logw_c, const int32_t* n_kept, int32_t capacity,
                             float delta, float eps0, ebd_range_mode range_mode, const float* y,
                             const float* lse, const float* var_hat, const float* b_t,
                             const float* radius) {
  if (dtype != EBD_F32 && dtype != EBD_BF16) return EBD_ERR_INVALID;
  if (batch < 1 || n_kv_heads < 1 || group < 1 || capacity < 1) return EBD_ERR_INVALID;
  if (!Q || !K_c || !V_c || !logw_c || !n_kept || !y || !lse || !var_hat || !b_t || !radius)
    return EBD_ERR_INVALID;
  if (!(delta > 0.f && delta < 1.f) || !(eps0 >= 0.f)) return EBD_ERR_INVALID;
  if (range_mode != EBD_RANGE_BOUND && range_mode != EBD_RANGE_EXACT) return EBD_ERR_INVALID;
  if (head_dim != 64 && head_dim != 128) return EBD_ERR_UNSUPPORTED;
  if (group > 2 * kSliceHeads) return EBD_ERR_UNSUPPORTED;
  const long long units = (long long)batch * n_kv_heads;
  if (units * group > 0x7fffffffLL || units > 65535) return EBD_ERR_UNSUPPORTED;
  return EBD_OK;
}

}  // namespace ebd

extern "C" ebd_status ebd_certified_decode(ebd_dtype dtype, int32_t batch, int32_t n_kv_heads,
                                           int32_t group, int32_t head_dim, const void* Q,
                                           const void* K_c, const void* V_c, const float* logw_c,
                                           const int32_t* n_kept, int32_t capacity, float delta,
                                           float eps0, ebd_range_mode range_mode, float* y,
                                           float* lse, float* var_hat, float* b_t, float* radius,
                                           int32_t* dev_status, void* workspace, size_t ws_bytes,
                                           void* stream) {
  const ebd_status arg = check_decode_args(dtype, batch, n_kv_heads, group, head_dim, Q, K_c,
                                           V_c, logw_c, n_kept, capacity, delta, eps0,
                                           range_mode, y, lse, var_hat, b_t, radius);
  if (arg != EBD_OK) return arg;
  const long long units = (long long)batch * n_kv_heads;
  const DecodePlan plan = plan_decode(dtype, batch, n_kv_heads, group, head_dim, capacity);
  if (!workspace || ws_bytes < plan.ws_bytes) return EBD_ERR_CAPACITY;
  cudaStream_t s = (cudaStream_t)stream;
  const size_t esize = dtype == EBD_F32 ? 4 : 2;

  DecodeArgs a;
  a.Kc = K_c;
  a.Vc = V_c;
  a.logw = logw_c;
  a.n_kept = n_kept;
  a.cap = capacity;
  a.n_kv_heads = n_kv_heads;
  a.gstride = group;
  a.splits = plan.splits;
  a.tokens_per_split = plan.tokens_per_split;
  a.part = (float*)workspace;
  a.dev_status = dev_status;

  ReduceArgs r;
  r.part = (const float*)workspace;
  r.Vc = V_c;
  r.n_kept = n_kept;
  r.cap = capacity;
  r.splits = plan.splits;
  r.gstride = group;
  r.log_inv_delta = logf(1.f / delta);
  r.eps0 = eps0;
  r.exact = range_mode == EBD_RANGE_EXACT;

  // one pass per slice of at most kSliceHeads query heads (one slice for G <= 8);
  // the slices run in stream order and reuse the workspace
  const int slices = decode_slices(group);
  for (int sl = 0; sl < slices; ++sl) {
    const int h0 = sl * group / slices, h1 = (sl + 1) * group / slices;
    a.group = r.group = h1 - h0;
    a.Q = static_cast<const char*>(Q) + (size_t)h0 * head_dim * esize;
    a.y = r.y = y + (size_t)h0 * head_dim;
    a.lse = r.lse = lse + h0;
    r.var = var_hat + h0;
    a.b_t = r.b_t = b_t + h0;
    r.radius = radius + h0;
    const int n_heads = (int)(units * a.group);
    ebd_status st;
    if (plan.fast && fast_decode_usable(a, r, (int)units)) {
      st = launch_fast_decode(dtype, head_dim, plan, a, r, (int)units, workspace, s);
    } else {
      st = dispatch_generic(false, dtype, head_dim, a, (int)units, s);
      if (st == EBD_OK) {
        const int rblocks = (n_heads + kReduceWarps - 1) / kReduceWarps;
        const dim3 rg(rblocks), rb(kReduceWarps * 32);
        if (dtype == EBD_F32) {
          if (head_dim == 128) decode_reduce_kernel<float, 128><<<rg, rb, 0, s>>>(r, n_heads);
          else decode_reduce_kernel<float, 64><<<rg, rb, 0, s>>>(r, n_heads);
        } else {
          if (head_dim == 128) decode_reduce_kernel<__nv_bfloat16, 128><<<rg, rb, 0, s>>>(r, n_heads);
          else decode_reduce_kernel<__nv_bfloat16, 64><<<rg, rb, 0, s>>>(r, n_heads);
        }
        st = launch_status();
      }
    }
    if (st != EBD_OK) return st;
    // exact range term: second pass over the slice's tail rows
    if (r.exact) {
      st = dispatch_generic(true, dtype, head_dim, a, (int)units, s);
      if (st != EBD_OK) return st;
    }
  }
  if (!r.exact) return EBD_OK;
  // the radius of every query head from its V_hat and exact range term
  r.group = r.gstride = group;
  r.y = y;
  r.lse = lse;
  r.var = var_hat;
  r.b_t = b_t;
  r.radius = radius;
  const int n_heads = (int)(units * group);
  const int warps = 4;
  if (head_dim == 128)
    decode_radius_kernel<128><<<(n_heads + warps - 1) / warps, warps * 32, 0, s>>>(r, n_heads);
  else
    decode_radius_kernel<64><<<(n_heads + warps - 1) / warps, warps * 32, 0, s>>>(r, n_heads);
  return launch_status();
}
