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
// come from the certified decode): on tensor cores for bf16 caches whose
// capacity is a multiple of 16, else one warp per token of a split.
#include <cuda_runtime.h>

#include "common.cuh"
#include "decode.cuh"
#include "internal.h"
#include "ptx.cuh"

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

// Tensor-core contributions (bf16, d in {64, 128}, G <= 8).  A warp takes a
// run of 16-token tiles of one unit, streamed by 16-byte cp.async into a
// 3-stage ring in the 128-byte-swizzled layout.  With tokens as the MMA's M
// and the query heads as its N (padded to 8), both products share one
// fragment layout: S^T = K Q^T (Q fragments in registers) and V Y^T (y_hat as
// bf16 hi + lo, about 16 bits), so each lane holds, for tokens g and g + 8
// (g = lane / 4) and heads 2q, 2q + 1 (q = lane % 4): the logit,
// v . (y_hat - c) and ||v - c||^2 from the same V fragments, c the unit's
// centring row (decode.cuh).  The contribution is
// (1 - pi) p^2 (||v - c||^2 - 2 (v - c).(y_hat - c) + ||y_hat - c||^2),
// p = 2^(x log2e - lse log2e): every term of the size of the values' spread,
// none of their common mean.  With a head column to spare (SPARE: G < 8) the
// product's column G carries c, so that ||v - c||^2 = ||v||^2 - 2 v.c + ||c||^2
// per token (exact products, a float32 cancellation of one token's terms);
// with G = 8 the V fragments are centred element by element.
constexpr int kCtmWarps = 8;
constexpr int kCtmTilesPerWarp = 16;
constexpr int kCtmStages = 3;

template <int D, bool SPARE>
__global__ void __launch_bounds__(kCtmWarps * 32)
    contrib_mma_kernel(const __nv_bfloat16* __restrict__ Q, const __nv_bfloat16* __restrict__ Kc,
                       const __nv_bfloat16* __restrict__ Vc, const float* __restrict__ logw,
                       const int32_t* __restrict__ n_kept, const float* __restrict__ y,
                       const float* __restrict__ lse, int group, int cap,
                       float* __restrict__ contrib) {
  constexpr int kBox = 16 * 128;                 // 16 rows x 128 B (64 columns)
  constexpr int kHalves = D / 64;
  constexpr int kTile = 2 * kHalves * kBox;      // K then V
  constexpr int CPR = D / 8;                     // 16-byte chunks per row
  constexpr int PER = 16 * CPR / 32;             // chunks per lane per tile (K or V)
  extern __shared__ unsigned char ctm_raw[];
  unsigned char* base = (unsigned char*)(((uintptr_t)ctm_raw + 1023) & ~(uintptr_t)1023);
  auto sm = reinterpret_cast<unsigned char(*)[kCtmStages][kTile]>(base);
  auto slw = reinterpret_cast<float(*)[kCtmStages][16]>(base + kCtmWarps * kCtmStages * kTile);
  const int unit = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, q = lane & 3;
  const int G = group;
  const int n = min(max(n_kept[unit], 0), cap);
  const int ntiles = (cap + 15) / 16;
  const int t_begin = (blockIdx.x * kCtmWarps + warp) * kCtmTilesPerWarp;
  if (t_begin >= ntiles) return;
  const int t_end = min(ntiles, t_begin + kCtmTilesPerWarp);
  const size_t hq0 = (size_t)unit * G;

  // the unit's centring row c (bf16, exact as a V row; zeros for an empty
  // unit): pairs at channels 16 kk + 2q (.x) and 16 kk + 8 + 2q (.y), the
  // channels of this lane's V fragments
  const int cr = centre_row(n);
  const __nv_bfloat16* crow = Vc + ((size_t)unit * cap + (cr < 0 ? 0 : cr)) * D;
  uint32_t cp[D / 16][2];  // -c, both bf16 halves negated
#pragma unroll
  for (int kk = 0; kk < D / 16; ++kk) {
    const uint32_t* c32 = reinterpret_cast<const uint32_t*>(crow + 16 * kk);
    cp[kk][0] = (cr < 0 ? 0u : c32[q]) ^ 0x80008000u;
    cp[kk][1] = (cr < 0 ? 0u : c32[4 + q]) ^ 0x80008000u;
  }
  // B fragments (k = d index, n = head): Q and y_hat - c (hi, lo) of head g;
  // with SPARE, column G carries c itself (bf16, exact: lo part 0)
  uint32_t qb[D / 16][2], yh[D / 16][2], yl[D / 16][2];
  {
    const bool hv = g < G;
    const bool cv = SPARE && g == G;
    const __nv_bfloat16* qrow = Q + (hq0 + (hv ? g : 0)) * D;
    const float* yrow = y + (hq0 + (hv ? g : 0)) * D;
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      const uint32_t* q32 = reinterpret_cast<const uint32_t*>(qrow + 16 * kk);
      qb[kk][0] = hv ? q32[q] : 0u;
      qb[kk][1] = hv ? q32[4 + q] : 0u;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const float y0 = hv ? yrow[16 * kk + 8 * h + 2 * q] + bf16_lo(cp[kk][h]) : 0.f;
        const float y1 = hv ? yrow[16 * kk + 8 * h + 2 * q + 1] + bf16_hi(cp[kk][h]) : 0.f;
        const uint32_t hi = pack_bf16(y0, y1);
        yh[kk][h] = cv ? cp[kk][h] ^ 0x80008000u : hi;
        yl[kk][h] = cv ? 0u : pack_bf16(y0 - bf16_lo(hi), y1 - bf16_hi(hi));
      }
    }
  }
  // per-head constants for the heads this lane's C fragments hold (2q, 2q + 1):
  // ||y_hat - c||^2 and c . (y_hat - c), by warp reductions
  float l2[2], yy[2] = {0.f, 0.f}, cy[2] = {0.f, 0.f}, cc = 0.f;
#pragma unroll
  for (int c = 0; c < 2; ++c) {
    const int h = 2 * q + c;
    l2[c] = h < G ? lse[hq0 + h] * kLog2e : 0.f;
  }
  for (int h = 0; h < G; ++h) {
    float s2 = 0.f, sc = 0.f;
#pragma unroll
    for (int e = lane; e < D; e += 32) {
      const float ce = cr < 0 ? 0.f : __bfloat162float(crow[e]);
      const float yc = y[(hq0 + h) * D + e] - ce;
      s2 = fmaf(yc, yc, s2);
      sc = fmaf(ce, yc, sc);
    }
    s2 = warp_sum(s2);
    sc = warp_sum(sc);
    if (h == 2 * q) { yy[0] = s2; cy[0] = sc; }
    if (h == 2 * q + 1) { yy[1] = s2; cy[1] = sc; }
  }
  if constexpr (SPARE) {  // ||c||^2
    float s2 = 0.f;
#pragma unroll
    for (int e = lane; e < D; e += 32) {
      const float ce = cr < 0 ? 0.f : __bfloat162float(crow[e]);
      s2 = fmaf(ce, ce, s2);
    }
    cc = warp_sum(s2);
  }
  const float kscale = kLog2e * rsqrtf((float)D);

  auto issue = [&](int t, int slot) {
    if (t < t_end) {
      const size_t row0 = (size_t)unit * cap + (size_t)t * 16;
      unsigned char* st = sm[warp][slot];
#pragma unroll
      for (int i = 0; i < PER; ++i) {
        const int c = lane + 32 * i;
        const int r = c / CPR, ch = c - r * CPR;
        const int off = (ch >> 3) * kBox + r * 128 + (((ch & 7) ^ (r & 7)) << 4);
        const size_t src = (row0 + r) * D + ch * 8;
        cp_async16(st + off, Kc + src);  // cap % 16 == 0: every row of the tile exists
        cp_async16(st + kHalves * kBox + off, Vc + src);
      }
      if (lane < 4) cp_async16(&slw[warp][slot][4 * lane], logw + row0 + 4 * lane);
    }
    cp_async_commit();
  };

#pragma unroll
  for (int p = 0; p < kCtmStages - 1; ++p) issue(t_begin + p, p);
  for (int t = t_begin; t < t_end; ++t) {
    const int slot = (t - t_begin) % kCtmStages;
    issue(t + kCtmStages - 1, (t - t_begin + kCtmStages - 1) % kCtmStages);
    cp_async_wait<kCtmStages - 1>();
    __syncwarp();
    const int tok0 = t * 16;
    const int nv = min(16, n - tok0);  // retained rows of this tile (<= 0: none)
    if (nv > 0) {
      const uint32_t kbase = smem_u32(sm[warp][slot]);
      const uint32_t vbase = kbase + kHalves * kBox;
      float st[4] = {0.f, 0.f, 0.f, 0.f}, vy[4] = {0.f, 0.f, 0.f, 0.f};
      float2 vn0 = make_float2(0.f, 0.f), vn1 = make_float2(0.f, 0.f);  // ||v - c||^2 of tokens g, g + 8
      const int tok = (lane & 7) + ((lane >> 3) & 1) * 8;
      const int csel = lane >> 4;
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const int chunk = 2 * kk + csel;
        const uint32_t off = (chunk >> 3) * kBox + tok * 128 + (((chunk & 7) ^ (tok & 7)) << 4);
        uint32_t a0, a1, a2, a3;
        ldsm_x4(kbase + off, a0, a1, a2, a3);
        mma_bf16_16816(st, a0, a1, a2, a3, qb[kk][0], qb[kk][1]);
        uint32_t v0, v1, v2, v3;
        ldsm_x4(vbase + off, v0, v1, v2, v3);
        mma_bf16_16816(vy, v0, v1, v2, v3, yh[kk][0], yh[kk][1]);
        mma_bf16_16816(vy, v0, v1, v2, v3, yl[kk][0], yl[kk][1]);
        // v0, v2 token g, v1, v3 token g + 8 (two bf16 each; channels
        // 16 kk + 2q (v0, v1) and 16 kk + 8 + 2q (v2, v3)): ||v||^2 (SPARE)
        // or ||v - c||^2
        float2 e0 = make_float2(bf16_lo(v0), bf16_hi(v0)), e2 = make_float2(bf16_lo(v2), bf16_hi(v2));
        float2 e1 = make_float2(bf16_lo(v1), bf16_hi(v1)), e3 = make_float2(bf16_lo(v3), bf16_hi(v3));
        if constexpr (!SPARE) {
          const float2 ca = make_float2(bf16_lo(cp[kk][0]), bf16_hi(cp[kk][0]));
          const float2 cb = make_float2(bf16_lo(cp[kk][1]), bf16_hi(cp[kk][1]));
          e0 = __fadd2_rn(e0, ca);
          e2 = __fadd2_rn(e2, cb);
          e1 = __fadd2_rn(e1, ca);
          e3 = __fadd2_rn(e3, cb);
        }
        vn0 = __ffma2_rn(e0, e0, __ffma2_rn(e2, e2, vn0));
        vn1 = __ffma2_rn(e1, e1, __ffma2_rn(e3, e3, vn1));
      }
      float vs0 = vn0.x + vn0.y, vs1 = vn1.x + vn1.y;
      vs0 += __shfl_xor_sync(0xffffffffu, vs0, 1);
      vs0 += __shfl_xor_sync(0xffffffffu, vs0, 2);
      vs1 += __shfl_xor_sync(0xffffffffu, vs1, 1);
      vs1 += __shfl_xor_sync(0xffffffffu, vs1, 2);
      if constexpr (SPARE) {
        // v.c of tokens g and g + 8 sits in column G: lane 4 g + G / 2
        const int src = 4 * g + (G >> 1);
        const float vc0 = __shfl_sync(0xffffffffu, (G & 1) ? vy[1] : vy[0], src);
        const float vc1 = __shfl_sync(0xffffffffu, (G & 1) ? vy[3] : vy[2], src);
        vs0 = vs0 - 2.f * vc0 + cc;  // ||v - c||^2
        vs1 = vs1 - 2.f * vc1 + cc;
      }
      // C fragment: st[0], st[1] = (token g, heads 2q, 2q+1); st[2], st[3] = (token g + 8, ...)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int r = g + (e >> 1) * 8;   // token in the tile
        const int h = 2 * q + (e & 1);    // query head
        if (r >= nv || h >= G) continue;
        const float lw = slw[warp][slot][r];
        const float p = exp2f(fmaf(st[e], kscale, fmaf(lw, kLog2e, -l2[e & 1])));
        const float vv = (e >> 1) ? vs1 : vs0;  // ||v - c||^2
        // (v - c).(y_hat - c) = v.(y_hat - c) - c.(y_hat - c)
        const float dist = fmaxf(0.f, vv - 2.f * (vy[e] - cy[e & 1]) + yy[e & 1]);
        const float omp = lw > 0.f ? one_minus_exp_neg(lw) : 0.f;
        contrib[(hq0 + h) * cap + tok0 + r] = omp * p * p * dist;
      }
    }
    // rows of this tile at or past n_kept (within capacity) get 0
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int r = g + (e >> 1) * 8, h = 2 * q + (e & 1);
      if (r >= max(nv, 0) && h < G && tok0 + r < cap) contrib[(hq0 + h) * cap + tok0 + r] = 0.f;
    }
    __syncwarp();  // every lane's reads of this stage are done before it is refilled
  }
  cp_async_wait<0>();
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
  if (capacity % 16 == 0 && aligned16(Q) && aligned16(K_c) && aligned16(V_c) &&
      aligned16(logw_c)) {
    const int ntiles = capacity / 16;
    const int per_cta = kCtmWarps * kCtmTilesPerWarp;
    const dim3 grid((ntiles + per_cta - 1) / per_cta, u);
    const int smem = kCtmWarps * kCtmStages * (2 * (head_dim / 64) * 16 * 128 + 16 * 4) + 1024;
    const bool spare = group < 8;
    auto kern = head_dim == 64 ? (spare ? contrib_mma_kernel<64, true> : contrib_mma_kernel<64, false>)
                               : (spare ? contrib_mma_kernel<128, true> : contrib_mma_kernel<128, false>);
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
        cudaSuccess)
      return EBD_ERR_CUDA;
    kern<<<grid, kCtmWarps * 32, smem, s>>>((const __nv_bfloat16*)Q, (const __nv_bfloat16*)K_c,
                                            (const __nv_bfloat16*)V_c, logw_c, n_kept, y, lse,
                                            group, capacity, contrib);
    return launch_status();
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
