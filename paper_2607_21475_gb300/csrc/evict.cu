// Eviction step of eviction-by-design on GB300 (sm_103a).
//
// Per (batch row b, KV head kvh) unit, one CTA of 1024 threads:
//   E1  certainty set A: protected positions (sinks, recency window) plus the
//       top-k_head unprotected tokens by score, equal scores to the lower index
//       (Section 3.3 and Appendix B of the paper).  Exact selection by an
//       MSB-first 8-bit radix select over order-preserving score keys; an
//       ordered scan among the tokens equal to the k-th key only when fewer of
//       them are needed than there are.
//   E2  inclusion probabilities on the tail T (Eq. 2): pi_i = clip(c s_i, eps, 1)
//       with c solving sum_T pi_i = m (clip-saturated tokens join A): bisection
//       on log c whose steps take the exact linear solve of the current
//       partition (clipped-high / linear / floor) when it lands in the bracket,
//       stopping once the partition reproduces its own solve.
//   E3  Poisson draw: keep_i = (u_i < pi_i), u_i from word i % 4 of Philox4x32-10
//       keyed by the seed at counter (i / 4, kvh, layer, b); or the systematic
//       design at the same pi (one uniform per unit, fixed-point cumulative sums).
//   E4  stable compaction: an ordered block scan of the keep flags writes the
//       token index and log(1/pi_i) of every kept token; a second, HBM-bound
//       kernel then copies the kept K and V rows with 16-byte loads.
// Two select kernels: up to 32768 tokens the unit's scores sit in shared
// memory (one float4 per thread per 4096-token group); beyond, they stay in
// global memory (L2-resident while the unit is worked on) and every pass reads
// them in 4096-token steps.  ebd_evict pipelines chunks of one SM count of
// units over streams so that the copy of one select wave overlaps the next.
// K, V and the scores may be page-locked host memory (read over the host link).
#include <cuda_runtime.h>
#include <float.h>
#include <math.h>
#include <stdint.h>

#include "common.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace ebd {

constexpr int kSelThreads = 1024;
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kMaxCtx = 1 << 20;

struct SelectArgs {
  const float* scores;  // [units, n_ctx]
  int n_ctx;            // row stride of scores (and pi_out, mask_out)
  const int32_t* n_len; // nullable [units]: context length of each unit (<= n_ctx)
  int n_kv_heads;
  int layer;
  uint64_t seed;
  int n_sink;
  int n_recent;
  int k_head;
  int budget;
  int iters;
  float eps;
  float* pi_out;        // nullable [units, N]
  uint8_t* mask_out;    // nullable [units, N]
  int32_t* idx_c;       // nullable [units, cap] (compaction outputs all set or all null)
  float* logw_c;        // [units, cap]
  int32_t* n_kept;      // [units]
  int cap;
  int32_t* dev_status;  // nullable
  int vec4;             // scores rows start 16-byte aligned (float4 loads)
  int systematic;       // tail design: 0 Poisson, 1 systematic at the same pi
  int unit0;            // first unit of this launch (CTA x handles unit unit0 + x)
};

enum PiMode : int { kPiFloor = 0, kPiAll = 1, kPiLinear = 2 };

// pi of a tail token, Eq. (2): min(1, max(eps, c s)).  The two saturated
// regimes are the same formula at an extreme c: a budget at or below the
// floor (every tail token at eps) is c = 0, and a budget that covers every
// positive score (those at 1, the rest at eps) is c = FLT_MAX, for which
// c s >= 1 at every normal s > 0.
__device__ __forceinline__ float tail_pi(float s, float c, float eps) {
  return fminf(1.f, fmaxf(eps, c * s));
}

__device__ __forceinline__ float saturated_c(int mode) { return mode == kPiAll ? FLT_MAX : 0.f; }

// One water-filling step of Eq. (2), taken by one thread.  Given the partition
// at the current scale c (nh tail tokens clipped at 1, nl at eps, the others
// summing to smid), narrow the bisection bracket [lo, hi] on log c and return
// the next c: the exact linear solve of this partition when it lies inside the
// bracket, else the bracket's midpoint.  `stop` is set once the partition
// reproduces its own solve (or the step no longer moves c).  float32
// throughout: the sums it takes are float32 partial sums, and on this GPU the
// fp64 pipe would make this serial step the longest part of an iteration.
__device__ __forceinline__ float water_fill_step(int m, int nh, int nl, float smid, float eps,
                                                 float c, float& lo, float& hi, int& stop) {
  const float gval = (float)nh + eps * (float)nl + c * smid;
  if (gval < (float)m) lo = fmaxf(lo, logf(c));
  else hi = fminf(hi, logf(c));
  const float clin = smid > 0.f ? ((float)(m - nh) - eps * (float)nl) / smid : -1.f;
  if (clin > 0.f && fabsf(clin - c) <= 1e-6f * c) {
    stop = 1;  // the partition at c reproduces its own solve
    return clin;
  }
  const float lcl = clin > 0.f ? logf(clin) : -INFINITY;
  const float next = (clin > 0.f && lcl > lo && lcl < hi) ? clin : expf(0.5f * (lo + hi));
  if (next == c) stop = 1;
  return next;
}

// ---------------------------------------------------------------------------
// Large contexts (N > 32768): the scores stay in global memory (L2-resident
// while the unit is worked on).  Every pass walks them in steps of 4096
// tokens, thread t taking tokens 4t .. 4t + 3 of a step (one float4 load; one
// Philox call gives the draws of all four), four steps per round so that four
// loads per thread are in flight.  The certainty set is a bit array in shared
// memory.  Passes: four radix digits (per-warp histograms for the first), the
// top-slice pass (with an ordered scan of the ties only when fewer of them are
// needed than there are), one stats pass, the water-filling solve of Eq. (2)
// (bisection steps replaced by the exact linear solve of the current partition
// when it lands in the bracket; 1-5 passes as a rule), one draw + compaction
// pass with one ordered scan per step.
// ---------------------------------------------------------------------------
constexpr int kBigStep = 4 * kSelThreads;  // tokens per step
constexpr int kBigUnroll = 4;              // steps per round

struct BigScratch {
  unsigned hist[256];
  int tot[kSelWarps];
  float rf[3][kSelWarps];
  int ri[2][kSelWarps];
  float c, lo, hi;  // solve state, updated by thread 0 only
  int stop;
  unsigned prefix, remaining, eqcount;
};

// Scores of tokens i0 .. i0 + 3 (0 at and past N); non-finite values read as 0
// and reported through `bad`; -0 folded onto +0.
__device__ __forceinline__ void load4(const float* s, int i0, int N, bool vec4, float (&v)[4],
                                      bool& bad) {
  if (vec4 && i0 + 3 < N) {
    const float4 t = __ldg(reinterpret_cast<const float4*>(s + i0));
    v[0] = t.x;
    v[1] = t.y;
    v[2] = t.z;
    v[3] = t.w;
  } else {
#pragma unroll
    for (int r = 0; r < 4; ++r) v[r] = i0 + r < N ? __ldg(s + i0 + r) : 0.f;
  }
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    if (!isfinite(v[r])) {
      bad = bad || (i0 + r < N);
      v[r] = 0.f;
    }
    v[r] += 0.0f;
  }
}

// Exclusive prefix over the block, in thread order, of `cnt`, and the block
// total; two barriers (sh.tot is free again when it returns).  T = unsigned
// sums modulo 2^32 (the systematic walk).
template <typename T>
__device__ __forceinline__ T big_scan(T cnt, T& total, BigScratch& sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  T incl = cnt;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const T n = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += n;
  }
  if (lane == 31) sh.tot[warp] = (int)incl;
  __syncthreads();
  T before = 0, tot = 0;
#pragma unroll 8
  for (int w = 0; w < kSelWarps; ++w) {
    const T c = (T)sh.tot[w];
    before += w < warp ? c : (T)0;
    tot += c;
  }
  __syncthreads();
  total = tot;
  return before + incl - cnt;
}

__global__ void __launch_bounds__(kSelThreads, 1) evict_select_kernel(SelectArgs a, int words_pad) {
  extern __shared__ uint32_t big_smem[];
  __shared__ BigScratch sh;
  uint32_t* cert_bits = big_smem;            // bit i set <=> token i in A
  unsigned* whist = big_smem + words_pad;    // [kSelWarps][256] first-digit histograms

  const int unit = a.unit0 + blockIdx.x;
  const int b = unit / a.n_kv_heads;
  const int kvh = unit - b * a.n_kv_heads;
  const int Nrow = a.n_ctx;
  const int N = a.n_len ? min(max(__ldg(a.n_len + unit), 0), Nrow) : Nrow;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float* s = a.scores + (size_t)unit * Nrow;
  const bool vec4 = a.vec4 != 0;
  const int ns = min(a.n_sink, N);
  const int rs = max(N - a.n_recent, 0);  // first protected trailing position
  const int n_prot = ns + (N - rs) - max(0, ns - rs);
  const int n_cand = N - n_prot;
  const int k = min(max(a.k_head, 0), n_cand);
  const float eps = a.eps;
  bool bad = false;
  auto cand = [&](int i) { return i < N && i >= ns && i < rs; };
  // the nibble of tokens i0 .. i0 + 3 (i0 % 4 == 0) in the certainty bits
  auto cert4 = [&](int i0) { return (cert_bits[i0 >> 5] >> (i0 & 31)) & 0xFu; };
  // the eight threads of a word combine their nibbles; one of them stores it
  auto put4 = [&](int i0, uint32_t n4, bool assign) {
    uint32_t v = n4 << (i0 & 31);
    v |= __shfl_xor_sync(0xffffffffu, v, 1);
    v |= __shfl_xor_sync(0xffffffffu, v, 2);
    v |= __shfl_xor_sync(0xffffffffu, v, 4);
    if ((lane & 7) == 0 && i0 < N) cert_bits[i0 >> 5] = assign ? v : (cert_bits[i0 >> 5] | v);
  };

  // protected positions
  for (int base = 0; base < N; base += kBigStep) {
    const int i0 = base + 4 * tid;
    uint32_t p4 = 0u;
#pragma unroll
    for (int r = 0; r < 4; ++r)
      if (i0 + r < N && !cand(i0 + r)) p4 |= 1u << r;
    put4(i0, p4, true);
  }
  __syncthreads();

  // ---- E1: top-k_head among the unprotected tokens ------------------------
  if (k > 0 && k < n_cand) {
    unsigned prefix = 0u, maskbits = 0u, remaining = (unsigned)k;
#pragma unroll 1
    for (int shift = 24; shift >= 0; shift -= 8) {
      for (int j = tid; j < 256; j += kSelThreads) sh.hist[j] = 0u;
      unsigned* wh = whist + warp * 256;
      if (shift == 24)
        for (int j = lane; j < 256; j += 32) wh[j] = 0u;
      __syncthreads();
#pragma unroll 1
      for (int base = 0; base < N; base += kBigStep * kBigUnroll) {
        float v[kBigUnroll][4];
#pragma unroll
        for (int q = 0; q < kBigUnroll; ++q)
          load4(s, base + q * kBigStep + 4 * tid, N, vec4, v[q], bad);
#pragma unroll
        for (int q = 0; q < kBigUnroll; ++q) {
          const int i0 = base + q * kBigStep + 4 * tid;
#pragma unroll
          for (int r = 0; r < 4; ++r) {
            if (!cand(i0 + r)) continue;
            const uint32_t key = orderable_key(v[q][r]);
            if (shift == 24) atomicAdd(&wh[key >> 24], 1u);
            else if ((key & maskbits) == prefix) atomicAdd(&sh.hist[(key >> shift) & 255u], 1u);
          }
        }
      }
      __syncthreads();
      if (shift == 24) {
        for (int j = tid; j < 256; j += kSelThreads) {
          unsigned t = 0u;
#pragma unroll 8
          for (int w = 0; w < kSelWarps; ++w) t += whist[w * 256 + j];
          sh.hist[j] = t;
        }
        __syncthreads();
      }
      if (warp == 0) {
        // lane L owns bins 255-8L .. 248-8L (descending key order)
        unsigned c[8];
        unsigned tot = 0;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          c[q] = sh.hist[255 - 8 * lane - q];
          tot += c[q];
        }
        unsigned incl = tot;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const unsigned n = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += n;
        }
        const unsigned excl = incl - tot;
        if (excl < remaining && incl >= remaining) {
          unsigned cum = excl;
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            if (cum + c[q] >= remaining) {
              sh.prefix = prefix | ((unsigned)(255 - 8 * lane - q) << shift);
              sh.remaining = remaining - cum;
              sh.eqcount = c[q];  // tokens whose key matches the prefix so far
              break;
            }
            cum += c[q];
          }
        }
      }
      __syncthreads();
      prefix = sh.prefix;
      remaining = sh.remaining;
      maskbits |= 255u << shift;
    }
    // prefix is the k-th largest key: every key above it joins A, and the
    // `remaining` lowest-index tokens equal to it (all of them, without an
    // ordered scan, when there are no more than that)
    const bool all_eq = sh.eqcount <= remaining;
    int taken = 0;
#pragma unroll 1
    for (int base = 0; base < N; base += kBigStep * kBigUnroll) {
      float v[kBigUnroll][4];
#pragma unroll
      for (int q = 0; q < kBigUnroll; ++q)
        load4(s, base + q * kBigStep + 4 * tid, N, vec4, v[q], bad);
#pragma unroll
      for (int q = 0; q < kBigUnroll; ++q) {
        const int i0 = base + q * kBigStep + 4 * tid;
        uint32_t gt4 = 0u, eq4 = 0u;
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          if (!cand(i0 + r)) continue;
          const uint32_t key = orderable_key(v[q][r]);
          if (key > prefix) gt4 |= 1u << r;
          else if (key == prefix) eq4 |= 1u << r;
        }
        uint32_t sel4 = gt4;
        if (all_eq) {
          sel4 |= eq4;
        } else {
          int total;
          int run = taken + big_scan(__popc(eq4), total, sh);
#pragma unroll
          for (int r = 0; r < 4; ++r) {
            if ((eq4 >> r) & 1u) {
              if (run < (int)remaining) sel4 |= 1u << r;
              ++run;
            }
          }
          taken += total;
        }
        put4(i0, sel4, false);
      }
    }
  } else if (k > 0) {  // every unprotected token is in the top slice
    const int words = (N + 31) >> 5;
    for (int wd = tid; wd < words; wd += kSelThreads) {
      unsigned m = 0xffffffffu;
      if (wd == words - 1 && (N & 31)) m = (1u << (N & 31)) - 1u;
      cert_bits[wd] = m;
    }
  }
  __syncthreads();

  // ---- E2: inclusion probabilities on the tail -----------------------------
  const int n_cert = n_prot + k;
  const int nT = N - n_cert;
  const int m = min(max(a.budget - n_cert, 0), nT);
  {
    float smax = -INFINITY, sminpos = INFINITY, spos = 0.f;
    int npos = 0;
#pragma unroll 1
    for (int base = 0; base < N; base += kBigStep * kBigUnroll) {
      float v[kBigUnroll][4];
#pragma unroll
      for (int q = 0; q < kBigUnroll; ++q)
        load4(s, base + q * kBigStep + 4 * tid, N, vec4, v[q], bad);
#pragma unroll
      for (int q = 0; q < kBigUnroll; ++q) {
        const int i0 = base + q * kBigStep + 4 * tid;
        const uint32_t c4 = i0 < N ? cert4(i0) : 0xFu;
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          if (i0 + r >= N || ((c4 >> r) & 1u)) continue;
          smax = fmaxf(smax, v[q][r]);
          if (v[q][r] > 0.f) {
            sminpos = fminf(sminpos, v[q][r]);
            spos += v[q][r];
            ++npos;
          }
        }
      }
    }
    smax = warp_max(smax);
    sminpos = warp_min(sminpos);
    npos = warp_sum(npos);
    spos = warp_sum(spos);
    if (lane == 0) {
      sh.rf[0][warp] = smax;
      sh.rf[1][warp] = sminpos;
      sh.rf[2][warp] = spos;
      sh.ri[0][warp] = npos;
    }
    __syncthreads();
    if (warp == 0) {
      float mx = sh.rf[0][lane], mn = sh.rf[1][lane];
      float sd = sh.rf[2][lane];
      int np = sh.ri[0][lane];
      mx = warp_max(mx);
      mn = warp_min(mn);
      sd = warp_sum(sd);
      np = warp_sum(np);
      if (lane == 0) {
        // scalar decisions once, by thread 0, and broadcast
        int md = kPiLinear;
        if (nT == 0 || (float)m <= eps * (float)nT) md = kPiFloor;
        else if ((float)m >= (float)np + eps * (float)(nT - np)) md = kPiAll;
        sh.stop = md != kPiLinear;
        if (md == kPiLinear) {
          sh.lo = logf(eps / mx);
          sh.hi = logf(1.f / mn);
          sh.c = fminf(fmaxf((float)m / sd, expf(sh.lo)), expf(sh.hi));
        } else {
          sh.c = saturated_c(md);
        }
      }
    }
    __syncthreads();
  }
  float c = sh.c;
#pragma unroll 1
  for (int it = 0; it < a.iters && !sh.stop; ++it) {
    int nhi = 0, nlo = 0;
    float smid = 0.f;
#pragma unroll 1
    for (int base = 0; base < N; base += kBigStep * kBigUnroll) {
      float v[kBigUnroll][4];
#pragma unroll
      for (int q = 0; q < kBigUnroll; ++q)
        load4(s, base + q * kBigStep + 4 * tid, N, vec4, v[q], bad);
#pragma unroll
      for (int q = 0; q < kBigUnroll; ++q) {
        const int i0 = base + q * kBigStep + 4 * tid;
        const uint32_t c4 = i0 < N ? cert4(i0) : 0xFu;
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          if (i0 + r >= N || ((c4 >> r) & 1u)) continue;
          const float t = c * v[q][r];
          if (t >= 1.f) ++nhi;
          else if (t <= eps) ++nlo;
          else smid += v[q][r];
        }
      }
    }
    nhi = warp_sum(nhi);
    nlo = warp_sum(nlo);
    smid = warp_sum(smid);
    // (the barrier closing the previous iteration ordered its reads of sh)
    if (lane == 0) {
      sh.ri[0][warp] = nhi;
      sh.ri[1][warp] = nlo;
      sh.rf[0][warp] = smid;
    }
    __syncthreads();
    if (warp == 0) {
      float sd = sh.rf[0][lane];
      int ah = sh.ri[0][lane], al = sh.ri[1][lane];
      sd = warp_sum(sd);
      ah = warp_sum(ah);
      al = warp_sum(al);
      if (lane == 0) {
        float lo = sh.lo, hi = sh.hi;
        int stop = 0;
        sh.c = water_fill_step(m, ah, al, sd, eps, c, lo, hi, stop);
        sh.stop = stop;
        sh.lo = lo;
        sh.hi = hi;
      }
    }
    __syncthreads();
    c = sh.c;
  }

  // ---- E3 + E4a: draws, stable compaction of (index, log 1/pi) -------------
  const bool compact = a.n_kept != nullptr;
  const bool systematic = compact && a.systematic;
  int kept = 0;
  // Systematic design (as in the shared-memory kernel): the tail in token
  // order, pi in units of 2^-32 (rounded to the nearest unit; pi = 1 adds 0
  // and is always kept), one uniform u per unit at counter word 0 = 2^32 - 1;
  // a tail token is kept when the running fraction of C - u carries out.
  // `frac`: that fraction before the current step (sums modulo 2^32).
  uint32_t frac = 0u;
  if (systematic) frac = 0u - ((draw_block(a.seed, a.layer, b, kvh, -1).x >> 8) << 8);
#pragma unroll 1
  for (int base = 0; base < N; base += kBigStep * kBigUnroll) {
    float v[kBigUnroll][4];
#pragma unroll
    for (int q = 0; q < kBigUnroll; ++q)
      load4(s, base + q * kBigStep + 4 * tid, N, vec4, v[q], bad);
#pragma unroll
    for (int q = 0; q < kBigUnroll; ++q) {
      const int i0 = base + q * kBigStep + 4 * tid;
      const uint32_t c4 = i0 < N ? cert4(i0) : 0xFu;
      uint4 w = make_uint4(0u, 0u, 0u, 0u);
      if (compact && !systematic && i0 < N) w = draw_block(a.seed, a.layer, b, kvh, i0 >> 2);
      const uint32_t wr[4] = {w.x, w.y, w.z, w.w};
      float pis[4];
      uint32_t keep4 = 0u, tail4 = 0u, units4[4] = {0u, 0u, 0u, 0u}, tsum = 0u;
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const int i = i0 + r;
        pis[r] = 1.f;
        if (i >= N) continue;
        const bool ct = (c4 >> r) & 1u;
        const float pi = ct ? 1.f : tail_pi(v[q][r], c, eps);
        pis[r] = pi;
        if (a.pi_out) a.pi_out[(size_t)unit * Nrow + i] = pi;
        if (a.mask_out) a.mask_out[(size_t)unit * Nrow + i] = ct ? 1 : 0;
        if (systematic) {
          if (ct) {
            keep4 |= 1u << r;
          } else {
            tail4 |= 1u << r;
            units4[r] = pi >= 1.f ? 0u : __float2uint_rn(pi * 4294967296.f);
            tsum += units4[r];
          }
        } else if (compact && (ct || word_to_uniform(wr[r]) < pi)) {
          keep4 |= 1u << r;
        }
      }
      if (systematic) {
        uint32_t stotal;
        uint32_t run = frac + big_scan<uint32_t>(tsum, stotal, sh);
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          if (!((tail4 >> r) & 1u)) continue;
          const uint32_t before = run;
          run += units4[r];
          if (pis[r] >= 1.f || run < before) keep4 |= 1u << r;  // a carry: an integer crossed
        }
        frac += stotal;
      }
      if (compact) {
        int total;
        int p = kept + big_scan<int>(__popc(keep4), total, sh);
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          if (!((keep4 >> r) & 1u)) continue;
          if (p < a.cap) {
            a.idx_c[(size_t)unit * a.cap + p] = i0 + r;
            a.logw_c[(size_t)unit * a.cap + p] = pis[r] >= 1.f ? 0.f : -logf(pis[r]);
          }
          ++p;
        }
        kept += total;
      }
    }
  }
  if (compact && tid == 0) {
    a.n_kept[unit] = kept;
    if (kept > a.cap) raise_status(a.dev_status, EBD_DEV_CAPACITY);
  }
  if (__syncthreads_or(bad) && tid == 0) raise_status(a.dev_status, EBD_DEV_NONFINITE);
}

// ---------------------------------------------------------------------------
// Shared-memory variant for N <= 4096 * JG (JG <= 8, i.e. N <= 32768).
// 1024 threads; thread t owns tokens g*4096 + 4t + r (g < JG, r < 4): the four
// tokens that share one Philox call live in one thread, and its scores sit in
// shared memory as one float4 per group (read once from HBM).  Membership is
// a 32-bit mask per thread (bit 4g + r).  Loops over groups stay rolled so the
// kernel stays small in the instruction cache.
// The top slice is an MSB-first radix select over 8-bit digits of the
// order-preserving keys: the load builds the first digit's histogram, one
// pass over every candidate settles the first digit (and builds the second
// digit's histogram), and later passes touch only the tokens still in
// contention.  A token leaves contention either into the top slice or into
// the tail, and the tail statistics that Eq. (2) starts from are taken as it
// leaves, so no separate pass gathers them.
// The scale c of Eq. (2) is found by bisection on log c whose steps are
// replaced by the exact linear solve inside the current partition whenever
// that solve lands inside the bracket (water-filling); it stops once the
// partition reproduces its own solve, after at most `iters` evaluations.
// ---------------------------------------------------------------------------
constexpr int kRegThreads = 1024;
constexpr int kRegWarps = kRegThreads / 32;
constexpr int kRegMaxGroups = 8;
constexpr int kGroupTokens = 4 * kRegThreads;
// Per-warp histograms sit 257 words apart, so that the lanes of the reduce,
// which read one bin from four warps' histograms at once, hit distinct banks.
constexpr int kHistStride = 257;

struct RegScratch {
  long long ll[kRegWarps];  // systematic design: per-warp prefix totals
  unsigned hist[256];
  int tot[kRegMaxGroups][kRegWarps];
  int off[kRegMaxGroups][kRegWarps];
  float rf[3][kRegWarps];
  int ri[2][kRegWarps];
  float res_f[3];
  int res_i[2];
  float c, lo, hi;  // solve state, updated by thread 0 only
  int stop;
  unsigned prefix, remaining, eqcount;
  int total;
  // published for the other CTAs of a unit's cluster (two buffers: an
  // exchange reuses the buffer of the one before the last)
  unsigned hist_x[2][256];
  float xf[2][3];
  int xi[2][2];
  int xres[2];
};

// Cross-warp combine of per-warp partials written to sh.rf / sh.ri by lane 0
// of every warp: warp 0 reduces the kRegWarps entries and publishes res_*.
// Callers bracket it with barriers.
__device__ __forceinline__ void combine_stats(RegScratch& sh) {
  const int lane = threadIdx.x & 31;
  if ((threadIdx.x >> 5) == 0) {
    float mx = sh.rf[0][lane], mn = sh.rf[1][lane], sd = sh.rf[2][lane];
    int n = sh.ri[0][lane];
    mx = warp_max(mx);
    mn = warp_min(mn);
    sd = warp_sum(sd);
    n = warp_sum(n);
    if (lane == 0) {
      sh.res_f[0] = mx;
      sh.res_f[1] = mn;
      sh.res_f[2] = sd;
      sh.res_i[0] = n;
    }
  }
}

__device__ __forceinline__ void combine_partition(RegScratch& sh) {
  const int lane = threadIdx.x & 31;
  if ((threadIdx.x >> 5) == 0) {
    float sd = sh.rf[0][lane];
    int a = sh.ri[0][lane], b = sh.ri[1][lane];
    sd = warp_sum(sd);
    a = warp_sum(a);
    b = warp_sum(b);
    if (lane == 0) {
      sh.res_f[2] = sd;
      sh.res_i[0] = a;
      sh.res_i[1] = b;
    }
  }
}

// Per-group counts of the set bits of `flags` (group g = bits 4g .. 4g + 3),
// one byte per group: groups 0-3 in `lo`, groups 4-7 in `hi`.
__device__ __forceinline__ void group_counts(uint32_t flags, uint32_t& lo, uint32_t& hi) {
  uint32_t x = flags - ((flags >> 1) & 0x55555555u);
  x = (x & 0x33333333u) + ((x >> 2) & 0x33333333u);  // each nibble holds its count
  uint32_t l = x & 0xFFFFu, h = x >> 16;
  l = (l | (l << 8)) & 0x00FF00FFu;
  l = (l | (l << 4)) & 0x0F0F0F0Fu;
  h = (h | (h << 8)) & 0x00FF00FFu;
  h = (h | (h << 4)) & 0x0F0F0F0Fu;
  lo = l;
  hi = h;
}

__device__ __forceinline__ int group_byte(uint32_t lo, uint32_t hi, int g) {
  return (int)(((g < 4 ? lo : hi) >> (8 * (g & 3))) & 0xFFu);
}

// Ordered count of the set bits of `flags` (bit 4g + r <-> token
// g*4096 + 4*tid + r).  One warp scan of the packed per-group counts (a warp's
// count in one group is at most 128, so the bytes never carry) gives every
// lane its exclusive prefix in all groups at once (`below_lo`, `below_hi`);
// afterwards sh.off[g][w] is the number of set bits at tokens before warp w's
// slice of group g.  Returns the block total.  The rank of a token is
// sh.off[g][warp] + group_byte(below, g) + its rank within the thread's group.
__device__ __forceinline__ int ordered_scan(uint32_t flags, int JG, RegScratch& sh,
                                            uint32_t& below_lo, uint32_t& below_hi) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t lo, hi;
  group_counts(flags, lo, hi);
  uint32_t il = lo, ih = hi;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t nl = __shfl_up_sync(0xffffffffu, il, o);
    const uint32_t nh = __shfl_up_sync(0xffffffffu, ih, o);
    if (lane >= o) {
      il += nl;
      ih += nh;
    }
  }
  below_lo = il - lo;
  below_hi = ih - hi;
  const uint32_t tl = __shfl_sync(0xffffffffu, il, 31);
  const uint32_t th = __shfl_sync(0xffffffffu, ih, 31);
  __syncthreads();  // previous readers of sh.tot / sh.off / sh.total are done
  if (lane < JG) sh.tot[lane][warp] = group_byte(tl, th, lane);
  __syncthreads();
  if (warp == 0) {
    const int E = JG * kRegWarps;               // <= 256
    const int PER = (E + 31) / 32;              // <= 8
    int local = 0;
#pragma unroll 1
    for (int q = 0; q < PER; ++q) {
      const int e = lane * PER + q;
      if (e < E) local += sh.tot[e / kRegWarps][e % kRegWarps];
    }
    int incl = local;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int n = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += n;
    }
    int run = incl - local;
#pragma unroll 1
    for (int q = 0; q < PER; ++q) {
      const int e = lane * PER + q;
      if (e < E) {
        const int v = sh.tot[e / kRegWarps][e % kRegWarps];
        sh.off[e / kRegWarps][e % kRegWarps] = run;
        run += v;
      }
    }
    if (lane == 31) sh.total = incl;
  }
  __syncthreads();
  return sh.total;
}

// Exclusive prefix over the ranks of a unit's cluster of a per-CTA count `v`
// (the same in every thread of the CTA), and the cluster total; every thread
// gets both.  Without a cluster (C == 1) that is (0, v).
__device__ __forceinline__ int cluster_scan(int v, RegScratch& sh, int C, int crank, int& xpar,
                                            int& total) {
  if (C == 1) {
    total = v;
    return 0;
  }
  if (threadIdx.x == 0) sh.xi[xpar][0] = v;
  cluster_barrier();
  if (threadIdx.x == 0) {
    const uint32_t addr = smem_u32(&sh.xi[xpar][0]);
    unsigned below = 0u, tot = 0u;  // unsigned: the systematic walk sums modulo 2^32
    for (int q = 0; q < C; ++q) {
      const unsigned x = ld_cluster_u32(cluster_map(addr, (uint32_t)q));
      if (q < crank) below += x;
      tot += x;
    }
    sh.xres[0] = (int)below;
    sh.xres[1] = (int)tot;
  }
  __syncthreads();
  xpar ^= 1;
  total = sh.xres[1];
  return sh.xres[0];
}

// One radix-select step: the per-warp histograms of the current digit are
// summed into sh.hist (over every CTA of the unit's cluster when C > 1), then
// warp 0 finds, from
// the top, the digit value holding the `remaining`-th largest key still in
// contention and publishes it (sh.prefix), the rank left inside it
// (sh.remaining) and its count (sh.eqcount).  Three barriers.
__device__ __forceinline__ void choose_digit(const unsigned* whist, RegScratch& sh,
                                             unsigned remaining, int C, int dpar) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  __syncthreads();  // every per-warp histogram is complete
  {
    // warp w sums bins 8w .. 8w + 7: lane l takes bin 8w + (l & 7) over warps
    // 8(l >> 3) .. 8(l >> 3) + 7, then four lanes combine by shuffles
    const int j = 8 * warp + (lane & 7), q = lane >> 3;
    unsigned t = 0u;
#pragma unroll
    for (int w = 0; w < kRegWarps / 4; ++w) t += whist[(q * (kRegWarps / 4) + w) * kHistStride + j];
    t += __shfl_xor_sync(0xffffffffu, t, 8);
    t += __shfl_xor_sync(0xffffffffu, t, 16);
    if (lane < 8) (C > 1 ? sh.hist_x[dpar][j] : sh.hist[j]) = t;
  }
  if (C > 1) {
    // the cluster's histogram: every CTA sums all CTAs' histograms
    cluster_barrier();
    if (tid < 256) {
      const uint32_t addr = smem_u32(&sh.hist_x[dpar][tid]);
      unsigned t = 0u;
      for (int q = 0; q < C; ++q) t += ld_cluster_u32(cluster_map(addr, (uint32_t)q));
      sh.hist[tid] = t;
    }
  }
  __syncthreads();
  if (warp == 0) {
    unsigned c[8];
    unsigned tot = 0;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      c[q] = sh.hist[255 - 8 * lane - q];
      tot += c[q];
    }
    unsigned incl = tot;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned n = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += n;
    }
    const unsigned excl = incl - tot;
    if (excl < remaining && incl >= remaining) {
      unsigned cum = excl;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        if (cum + c[q] >= remaining) {
          sh.prefix = (unsigned)(255 - 8 * lane - q);  // the chosen digit
          sh.remaining = remaining - cum;
          sh.eqcount = c[q];  // keys in contention with this digit
          break;
        }
        cum += c[q];
      }
    }
  }
  __syncthreads();
}

// 1024 threads of at most 56 registers (57,344 of the SM's 65,536) leave room
// for one 128-thread gather CTA beside a select CTA in the pipelined eviction.
__global__ void __maxnreg__(56) evict_select_smem_kernel(SelectArgs a, int JG) {
  extern __shared__ float4 s4[];  // [JG][1024]: scores of thread t, group g at s4[g*1024 + t]
  // followed by the per-warp radix histograms [kRegWarps][kHistStride]
  unsigned* whist = reinterpret_cast<unsigned*>(s4 + JG * kRegThreads);
  __shared__ RegScratch sh;
  const float* sflat = reinterpret_cast<const float*>(s4);
  const int C = (int)cluster_size();      // CTAs per unit: 1 without a cluster launch
  const int crank = (int)cluster_rank();  // this CTA's slice of the unit
  const int unit = a.unit0 + (int)blockIdx.x / C;
  const int b = unit / a.n_kv_heads;
  const int kvh = unit - b * a.n_kv_heads;
  const int Nrow = a.n_ctx;
  const int N = a.n_len ? min(max(__ldg(a.n_len + unit), 0), Nrow) : Nrow;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float* sp = a.scores + (size_t)unit * Nrow;
  const int ns = min(a.n_sink, N);
  const int rs = max(N - a.n_recent, 0);
  const int n_prot = ns + (N - rs) - max(0, ns - rs);
  const int n_cand = N - n_prot;
  const int k = min(max(a.k_head, 0), n_cand);
  const float eps = a.eps;
  const bool radix = k > 0 && k < n_cand;
  unsigned* wh = whist + warp * kHistStride;
  const int t0 = crank * JG * kGroupTokens;  // first token of this CTA's slice
  auto ltok = [&](int g, int r) { return g * kGroupTokens + 4 * tid + r; };  // within the slice
  auto tok = [&](int g, int r) { return t0 + ltok(g, r); };
  int xpar = 0;  // cluster exchange buffer (cluster-uniform)
  auto is_cand = [&](int i) { return i >= ns && i < rs; };  // for i < N
  auto score_of = [&](int bitpos) {  // bit 4g + r of the membership masks
    return sflat[((bitpos >> 2) * kRegThreads + tid) * 4 + (bitpos & 3)];
  };
  auto zero_hist = [&]() {
    for (int j = lane; j < 256; j += 32) wh[j] = 0u;
    __syncwarp();
  };

  // statistics of the tail tokens this thread has met (the start of Eq. 2)
  float smax = -INFINITY, sminpos = INFINITY, spos = 0.f;
  int npos = 0;
  auto add_tail = [&](float v) {
    smax = fmaxf(smax, v);
    if (v > 0.f) {
      sminpos = fminf(sminpos, v);
      spos += v;
      ++npos;
    }
  };

  // ---- load: sanitise, fold -0 onto +0, protected positions -------------------
  // every group's load is issued before the first is used
  if (radix) zero_hist();
  bool bad = false;
  uint32_t cert = 0u, valid = 0u;
  float4 raw[kRegMaxGroups];
#pragma unroll
  for (int g = 0; g < kRegMaxGroups; ++g) {
    raw[g] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (g < JG) {
      const int i0 = tok(g, 0);
      if (a.vec4 && i0 + 3 < N) {
        raw[g] = __ldg(reinterpret_cast<const float4*>(sp + i0));
      } else {
        if (i0 < N) raw[g].x = __ldg(sp + i0);
        if (i0 + 1 < N) raw[g].y = __ldg(sp + i0 + 1);
        if (i0 + 2 < N) raw[g].z = __ldg(sp + i0 + 2);
        if (i0 + 3 < N) raw[g].w = __ldg(sp + i0 + 3);
      }
    }
  }
#pragma unroll
  for (int g = 0; g < kRegMaxGroups; ++g) {
    if (g >= JG) break;
    float v[4] = {raw[g].x, raw[g].y, raw[g].z, raw[g].w};
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int i = tok(g, r);
      if (!isfinite(v[r])) {
        bad = bad || (i < N);
        v[r] = 0.f;
      }
      v[r] += 0.0f;
      if (i >= N) continue;
      const uint32_t bit = 1u << (4 * g + r);
      valid |= bit;
      if (!is_cand(i)) cert |= bit;  // protected
      else if (radix) atomicAdd(&wh[orderable_key(v[r]) >> 24], 1u);  // first digit
      else if (k == 0) add_tail(v[r]);  // no top slice: every candidate is tail
    }
    s4[g * kRegThreads + tid] = make_float4(v[0], v[1], v[2], v[3]);
  }

  // ---- E1: top-k_head among the unprotected tokens ------------------------
  if (radix) {
    uint32_t live = valid & ~cert;  // candidates whose keys match the chosen digits
    unsigned remaining = (unsigned)k;
    bool done = false;
#pragma unroll 1
    for (int shift = 24;; shift -= 8) {
      choose_digit(whist, sh, remaining, C, (shift >> 3) & 1);
      const unsigned digit = sh.prefix;
      remaining = sh.remaining;
      done = sh.eqcount == remaining;  // every key with this digit is in the slice
      const bool last = done || shift == 0;
      const int nshift = last ? 0 : shift - 8;
      if (!last) zero_hist();
      // a token with a higher digit joins the slice, a lower one the tail; an
      // equal one stays in contention and counts toward the next digit
      auto settle = [&](int bitpos, float v) {
        const uint32_t key = orderable_key(v);
        const unsigned d = (key >> shift) & 255u;
        const uint32_t bit = 1u << bitpos;
        if (d > digit || (d == digit && done)) {
          cert |= bit;
          live &= ~bit;
        } else if (d < digit) {
          live &= ~bit;
          add_tail(v);
        } else if (!last) {
          atomicAdd(&wh[(key >> nshift) & 255u], 1u);
        }
      };
      if (shift == 24) {
        // every candidate is still in contention
#pragma unroll 1
        for (int g = 0; g < JG; ++g) {
          const uint32_t l4 = (live >> (4 * g)) & 0xFu;
          if (!l4) continue;
          const float4 v4 = s4[g * kRegThreads + tid];
          const float vv[4] = {v4.x, v4.y, v4.z, v4.w};
#pragma unroll
          for (int r = 0; r < 4; ++r)
            if ((l4 >> r) & 1u) settle(4 * g + r, vv[r]);
        }
      } else {
        for (uint32_t m = live; m; m &= m - 1) {
          const int bitpos = __ffs(m) - 1;
          settle(bitpos, score_of(bitpos));
        }
      }
      if (last) break;
    }
    if (!done) {
      // `live` holds the tokens whose key equals the k-th largest, more of
      // them than are needed: the `remaining` lowest-index ones join the slice
      uint32_t bl, bh;
      int ties_all;
      const int lower = cluster_scan(ordered_scan(live, JG, sh, bl, bh), sh, C, crank, xpar, ties_all);
#pragma unroll 1
      for (int g = 0; g < JG; ++g) {
        const uint32_t e4 = (live >> (4 * g)) & 0xFu;
        if (!e4) continue;
        int run = lower + sh.off[g][warp] + group_byte(bl, bh, g);
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          if (!((e4 >> r) & 1u)) continue;
          if (run < (int)remaining) cert |= 1u << (4 * g + r);
          else add_tail(score_of(4 * g + r));
          ++run;
        }
      }
    }
  } else if (k > 0) {
    cert = valid;  // every unprotected token is in the top slice
  }
  const uint32_t tail = valid & ~cert;
  auto is_tail = [&](int g, int r) { return (tail >> (4 * g + r)) & 1u; };

  // ---- E2: inclusion probabilities on the tail ---------------------------
  const int n_cert = n_prot + k;
  const int nT = N - n_cert;
  const int m = min(max(a.budget - n_cert, 0), nT);
  smax = warp_max(smax);
  sminpos = warp_min(sminpos);
  npos = warp_sum(npos);
  spos = warp_sum(spos);
  __syncthreads();
  if (lane == 0) {
    sh.rf[0][warp] = smax;
    sh.rf[1][warp] = sminpos;
    sh.rf[2][warp] = spos;
    sh.ri[0][warp] = npos;
  }
  __syncthreads();
  combine_stats(sh);
  __syncthreads();
  if (C > 1) {
    // the cluster's statistics, combined in rank order (the same in every CTA)
    if (tid == 0) {
      sh.xf[xpar][0] = sh.res_f[0];
      sh.xf[xpar][1] = sh.res_f[1];
      sh.xf[xpar][2] = sh.res_f[2];
      sh.xi[xpar][0] = sh.res_i[0];
    }
    cluster_barrier();
    if (tid == 0) {
      float mx = -INFINITY, mn = INFINITY, sd = 0.f;
      int n = 0;
      for (int q = 0; q < C; ++q) {
        mx = fmaxf(mx, ld_cluster_f32(cluster_map(smem_u32(&sh.xf[xpar][0]), (uint32_t)q)));
        mn = fminf(mn, ld_cluster_f32(cluster_map(smem_u32(&sh.xf[xpar][1]), (uint32_t)q)));
        sd += ld_cluster_f32(cluster_map(smem_u32(&sh.xf[xpar][2]), (uint32_t)q));
        n += (int)ld_cluster_u32(cluster_map(smem_u32(&sh.xi[xpar][0]), (uint32_t)q));
      }
      sh.res_f[0] = mx;
      sh.res_f[1] = mn;
      sh.res_f[2] = sd;
      sh.res_i[0] = n;
    }
    xpar ^= 1;
  }
  // Scalar decisions are taken once, by thread 0, and broadcast.
  if (tid == 0) {
    const float smax_b = sh.res_f[0], sminpos_b = sh.res_f[1];
    const int npos_b = sh.res_i[0];
    int md = kPiLinear;
    if (nT == 0 || (float)m <= eps * (float)nT) md = kPiFloor;
    else if ((float)m >= (float)npos_b + eps * (float)(nT - npos_b)) md = kPiAll;
    sh.stop = md != kPiLinear;
    if (md == kPiLinear) {
      sh.lo = logf(eps / smax_b);
      sh.hi = logf(1.f / sminpos_b);
      sh.c = fminf(fmaxf((float)m / sh.res_f[2], expf(sh.lo)), expf(sh.hi));
    } else {
      sh.c = saturated_c(md);
    }
  }
  __syncthreads();
  float c = sh.c;
#pragma unroll 1
  for (int it = 0; it < a.iters && !sh.stop; ++it) {
    int nhi = 0, nlo = 0;
    float smid = 0.f;
#pragma unroll 1
    for (int g = 0; g < JG; ++g) {
      const float4 v4 = s4[g * kRegThreads + tid];
      const float vv[4] = {v4.x, v4.y, v4.z, v4.w};
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        if (!is_tail(g, r)) continue;
        const float t = c * vv[r];
        if (t >= 1.f) ++nhi;
        else if (t <= eps) ++nlo;
        else smid += vv[r];
      }
    }
    nhi = warp_sum(nhi);
    nlo = warp_sum(nlo);
    smid = warp_sum(smid);
    // (the barrier closing the previous iteration ordered its reads of sh)
    if (lane == 0) {
      sh.ri[0][warp] = nhi;
      sh.ri[1][warp] = nlo;
      sh.rf[0][warp] = smid;
    }
    __syncthreads();
    combine_partition(sh);
    if (C > 1) {
      if (tid == 0) {
        sh.xf[xpar][0] = sh.res_f[2];
        sh.xi[xpar][0] = sh.res_i[0];
        sh.xi[xpar][1] = sh.res_i[1];
      }
      cluster_barrier();
      if (tid == 0) {
        float sd = 0.f;
        int nh = 0, nl = 0;
        for (int q = 0; q < C; ++q) {
          sd += ld_cluster_f32(cluster_map(smem_u32(&sh.xf[xpar][0]), (uint32_t)q));
          nh += (int)ld_cluster_u32(cluster_map(smem_u32(&sh.xi[xpar][0]), (uint32_t)q));
          nl += (int)ld_cluster_u32(cluster_map(smem_u32(&sh.xi[xpar][1]), (uint32_t)q));
        }
        sh.res_f[2] = sd;
        sh.res_i[0] = nh;
        sh.res_i[1] = nl;
      }
      xpar ^= 1;
    }
    if (tid == 0) {
      float lo = sh.lo, hi = sh.hi;
      int stop = 0;
      sh.c = water_fill_step(m, sh.res_i[0], sh.res_i[1], sh.res_f[2], eps, c, lo, hi, stop);
      sh.stop = stop;
      sh.lo = lo;
      sh.hi = hi;
    }
    __syncthreads();
    c = sh.c;
  }

  if (a.pi_out || a.mask_out) {
#pragma unroll 1
    for (int g = 0; g < JG; ++g) {
      const float4 v4 = s4[g * kRegThreads + tid];
      const float vv[4] = {v4.x, v4.y, v4.z, v4.w};
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const int i = tok(g, r);
        if (!((valid >> (4 * g + r)) & 1u)) continue;
        const bool ct = (cert >> (4 * g + r)) & 1u;
        if (a.pi_out) a.pi_out[(size_t)unit * Nrow + i] = ct ? 1.f : tail_pi(vv[r], c, eps);
        if (a.mask_out) a.mask_out[(size_t)unit * Nrow + i] = ct ? 1 : 0;
      }
    }
  }
  // ---- E3 + E4a: draws and ordered compaction of (index, log 1/pi) --------
  const bool compact = a.n_kept != nullptr;
  uint32_t keep = cert;
  if (compact && a.systematic) {
    // Fixed-size systematic sampling at the same pi (Hajek 1964): the tail in
    // token order, cumulative sums C_i of pi in units of 2^-32 (each pi rounded
    // to the nearest unit), one uniform u per unit; token i is kept when an
    // integer lies in (C_{i-1} - u, C_i - u].  Only the fractional part of
    // C - u matters, so the walk adds pi_i (mod 2^32) to it and keeps the token
    // on a carry out (pi_i = 1: always).  Inclusion probability pi_i, tail size
    // floor or ceil of sum pi.  Warp w walks tokens [1024 w, 1024 w + 1024) in
    // rows of 32 (lane = consecutive token: conflict-free reads) with a warp
    // scan per row, after one block scan of the warps' totals.  Tail and keep
    // flags move to and from the load layout through two bit arrays in the
    // (now free) histogram scratch.
    const uint4 wu = draw_block(a.seed, a.layer, b, kvh, -1);  // counter word 0 = 2^32 - 1
    const uint32_t u32 = (wu.x >> 8) << 8;                     // u in units of 2^-32
    uint32_t* tailbits = whist;                                  // [kRegMaxGroups * 4096 / 32]
    uint32_t* keepbits = whist + kRegMaxGroups * kGroupTokens / 32;
    const int ntok = JG * kGroupTokens;
    const int nwords = ntok / 32;                                // == JG * 128 <= 1024
    if (tid < nwords) tailbits[tid] = 0u;
    __syncthreads();
#pragma unroll 1
    for (int g = 0; g < JG; ++g) {
      const uint32_t t4 = (tail >> (4 * g)) & 0xFu;
      const int i0 = ltok(g, 0);
      if (t4) atomicOr(&tailbits[i0 >> 5], t4 << (i0 & 31));
    }
    __syncthreads();
    auto score_at = [&](int i) {  // token i of the load layout
      return sflat[((i >> 12) * kRegThreads + ((i & 4095) >> 2)) * 4 + (i & 3)];
    };
    // pi in units of 2^-32 (mod 2^32: pi = 1 adds 0 to the fraction)
    auto units32 = [&](float sv, bool& full) {
      const float p = tail_pi(sv, c, eps);
      full = p >= 1.f;
      return full ? 0u : __float2uint_rn(p * 4294967296.f);
    };
    const int wbase = 1024 * warp;
    uint32_t part = 0u;
    if (wbase < ntok) {
#pragma unroll 4
      for (int j = 0; j < 32; ++j) {
        const int i = wbase + 32 * j + lane;
        bool full;
        if ((tailbits[i >> 5] >> lane) & 1u) part += units32(score_at(i), full);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
    if (lane == 0) sh.ll[warp] = (long long)part;
    __syncthreads();
    uint32_t cta_part = 0u;
#pragma unroll 8
    for (int w2 = 0; w2 < kRegWarps; ++w2) cta_part += (uint32_t)sh.ll[w2];
    int parts_all;
    // fractional part of C - u before this warp's tokens
    uint32_t frac = 0u - u32 + (uint32_t)cluster_scan((int)cta_part, sh, C, crank, xpar, parts_all);
#pragma unroll 8
    for (int w2 = 0; w2 < kRegWarps; ++w2) frac += w2 < warp ? (uint32_t)sh.ll[w2] : 0u;
    if (wbase < ntok) {
#pragma unroll 1
      for (int j = 0; j < 32; ++j) {
        const int i = wbase + 32 * j + lane;
        const bool is_t = (tailbits[i >> 5] >> lane) & 1u;
        bool full = false;
        const uint32_t v = is_t ? units32(score_at(i), full) : 0u;
        uint32_t incl = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t nb = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += nb;
        }
        const uint32_t after = frac + incl, before = after - v;
        const bool sel = is_t && (full || after < before);  // a carry: an integer crossed
        const uint32_t mk = __ballot_sync(0xffffffffu, sel);
        if (lane == 0) keepbits[i >> 5] = mk;
        frac += __shfl_sync(0xffffffffu, incl, 31);
      }
    }
    __syncthreads();
#pragma unroll 1
    for (int g = 0; g < JG; ++g) {
      const int i0 = ltok(g, 0);
      const uint32_t k4 = (keepbits[i0 >> 5] >> (i0 & 31)) & 0xFu;
      if (!k4) continue;
      keep |= k4 << (4 * g);
      float4& slot = s4[g * kRegThreads + tid];
      float vv[4] = {slot.x, slot.y, slot.z, slot.w};
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const float pi = tail_pi(vv[r], c, eps);
        if ((k4 >> r) & 1u) vv[r] = pi >= 1.f ? 0.f : -logf(pi);
      }
      slot = make_float4(vv[0], vv[1], vv[2], vv[3]);
    }
  } else if (compact) {
    // Poisson design: keep a tail token when its uniform falls below pi
#pragma unroll 1
    for (int g = 0; g < JG; ++g) {
      const uint32_t t4 = (tail >> (4 * g)) & 0xFu;
      if (!__any_sync(0xffffffffu, t4 != 0u)) continue;
      const uint4 w = draw_block(a.seed, a.layer, b, kvh, (t0 >> 2) + g * kRegThreads + tid);
      if (!t4) continue;
      float4& slot = s4[g * kRegThreads + tid];
      float vv[4] = {slot.x, slot.y, slot.z, slot.w};
      const uint32_t wr[4] = {w.x, w.y, w.z, w.w};
      uint32_t k4 = 0u;
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const float pi = tail_pi(vv[r], c, eps);
        if (((t4 >> r) & 1u) && word_to_uniform(wr[r]) < pi) {
          k4 |= 1u << r;
          vv[r] = pi >= 1.f ? 0.f : -logf(pi);  // the score is not needed again
        }
      }
      if (k4) {
        slot = make_float4(vv[0], vv[1], vv[2], vv[3]);
        keep |= k4 << (4 * g);
      }
    }
  }
  if (compact) {
    uint32_t bl, bh;
    int total;
    const int lower = cluster_scan(ordered_scan(keep, JG, sh, bl, bh), sh, C, crank, xpar, total);
    int32_t* idx_row = a.idx_c + (size_t)unit * a.cap;
    float* logw_row = a.logw_c + (size_t)unit * a.cap;
#pragma unroll 1
    for (int g = 0; g < JG; ++g) {
      // one store per kept token, group by group so that a warp's stores fall
      // close together
      int p = lower + sh.off[g][warp] + group_byte(bl, bh, g);
      for (uint32_t k4 = (keep >> (4 * g)) & 0xFu; k4; k4 &= k4 - 1, ++p) {
        const int bitpos = 4 * g + __ffs(k4) - 1;
        if (p < a.cap) {
          // a kept tail token's slot holds its log(1/pi) by now
          idx_row[p] = tok(g, bitpos & 3);
          logw_row[p] = ((cert >> bitpos) & 1u) ? 0.f : score_of(bitpos);
        }
      }
    }
    if (tid == 0 && crank == 0) {
      a.n_kept[unit] = total;
      if (total > a.cap) raise_status(a.dev_status, EBD_DEV_CAPACITY);
    }
  }
  if (__syncthreads_or(bad) && tid == 0) raise_status(a.dev_status, EBD_DEV_NONFINITE);
  if (C > 1) cluster_barrier();  // no CTA leaves while another may read its shared memory
}

// E4b: copy kept K and V rows (16-byte chunks, `cpr` chunks per row).
constexpr int kGatherThreads = 128;  // small CTAs also fit beside a select CTA
constexpr int kGatherUnroll = 4;

__global__ void __launch_bounds__(kGatherThreads) gather_rows_kernel(
    const uint4* __restrict__ K, const uint4* __restrict__ V, uint4* __restrict__ Kc,
    uint4* __restrict__ Vc, const int32_t* __restrict__ idx_c, const int32_t* __restrict__ n_kept,
    int n_ctx, int cap, int cpr, int unit0) {
  const int unit = unit0 + blockIdx.y;
  const int n = min(n_kept[unit], cap);
  const long long items = (long long)n * cpr;
  const long long stride = (long long)gridDim.x * kGatherThreads;
  const int32_t* idx = idx_c + (size_t)unit * cap;
  const size_t src_base = (size_t)unit * n_ctx * cpr;
  const size_t dst_base = (size_t)unit * cap * cpr;
  for (long long it0 = (long long)blockIdx.x * kGatherThreads + threadIdx.x; it0 < items;
       it0 += stride * kGatherUnroll) {
    uint4 kv[kGatherUnroll], vv[kGatherUnroll];
    size_t dst[kGatherUnroll];
    bool ok[kGatherUnroll];
#pragma unroll
    for (int u = 0; u < kGatherUnroll; ++u) {
      const long long it = it0 + u * stride;
      const bool live = it < items;
      ok[u] = false;
      if (live) {
        const int p = (int)(it / cpr);
        const int ch = (int)(it - (long long)p * cpr);
        const int r = idx[p];
        // a row whose index lies outside the context is read from row 0 and
        // not stored: the copy never reads out of bounds
        ok[u] = (unsigned)r < (unsigned)n_ctx;
        const size_t src = src_base + (size_t)(ok[u] ? r : 0) * cpr + ch;
        dst[u] = dst_base + (size_t)p * cpr + ch;
        kv[u] = __ldg(K + src);
        vv[u] = __ldg(V + src);
      }
    }
#pragma unroll
    for (int u = 0; u < kGatherUnroll; ++u) {
      if (ok[u]) {
        Kc[dst[u]] = kv[u];
        Vc[dst[u]] = vv[u];
      }
    }
  }
}

__global__ void philox_words_kernel(uint64_t seed, int layer, int n_kv_heads, int n_ctx,
                                    long long total, uint32_t* out) {
  for (long long t = (long long)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (long long)gridDim.x * blockDim.x) {
    const long long unit = t / n_ctx;
    const int i = (int)(t - unit * n_ctx);
    const int b = (int)(unit / n_kv_heads);
    const int kvh = (int)(unit - (long long)b * n_kv_heads);
    out[t] = draw_word(seed, layer, b, kvh, i);
  }
}

int sm_count() {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (dev < 0 || dev >= 64) return 148;
  if (!cached[dev]) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      n = 148;
    cached[dev] = n;
  }
  return cached[dev];
}

ebd_status check_design(const ebd_design* d) {
  if (!d) return EBD_ERR_INVALID;
  if (d->batch < 1 || d->n_kv_heads < 1 || d->n_ctx < 1 || d->n_ctx > kMaxCtx) return EBD_ERR_INVALID;
  if ((long long)d->batch * d->n_kv_heads > 0x7fffffffLL) return EBD_ERR_INVALID;
  if (d->n_sink < 0 || d->n_recent < 0 || d->k_head < 0 || d->budget_tokens < 0) return EBD_ERR_INVALID;
  if (d->bisect_iters < 1 || d->bisect_iters > 200) return EBD_ERR_INVALID;
  if (d->sampling != EBD_SAMPLING_POISSON && d->sampling != EBD_SAMPLING_SYSTEMATIC)
    return EBD_ERR_INVALID;
  if (!(d->eps > 0.f && d->eps <= 1.f)) return EBD_ERR_INVALID;
  return EBD_OK;
}

// CTAs per unit for the shared-memory select: as many as the unit's scores
// need (32768 tokens per CTA), then more, up to a cluster of 8, while the
// request would leave SMs idle and every CTA keeps at least 4096 tokens.
// 0: the context is too long for a cluster (the global-memory kernel takes it).
constexpr int kMaxSelectCluster = 8;
int select_cluster_size(int n_ctx, int units) {
  const int per_cta = kRegMaxGroups * kGroupTokens;
  const int need = (n_ctx + per_cta - 1) / per_cta;
  if (need > kMaxSelectCluster) return 0;
  int C = need;
  const long long sms = sm_count();
  while (2 * C <= kMaxSelectCluster && (long long)units * 2 * C <= sms &&
         n_ctx >= 2 * C * kGroupTokens)
    C *= 2;
  return C;
}

ebd_status launch_select_range(const ebd_design* d, const float* scores, const int32_t* n_len,
                               float* pi, uint8_t* mask, int32_t* idx_c, float* logw_c,
                               int32_t* n_kept, int cap, int32_t* dev_status, int unit0,
                               int n_units, cudaStream_t stream, int ctas_per_unit) {
  SelectArgs a;
  a.scores = scores;
  a.n_ctx = d->n_ctx;
  a.n_len = n_len;
  a.n_kv_heads = d->n_kv_heads;
  a.layer = d->layer;
  a.seed = d->seed;
  a.n_sink = d->n_sink;
  a.n_recent = d->n_recent;
  a.k_head = d->k_head;
  a.budget = d->budget_tokens;
  a.iters = d->bisect_iters;
  a.eps = d->eps;
  a.pi_out = pi;
  a.mask_out = mask;
  a.idx_c = idx_c;
  a.logw_c = logw_c;
  a.n_kept = n_kept;
  a.cap = cap;
  a.dev_status = dev_status;
  a.vec4 = (((uintptr_t)scores & 15u) == 0 && (d->n_ctx & 3) == 0) ? 1 : 0;
  a.systematic = d->sampling == EBD_SAMPLING_SYSTEMATIC ? 1 : 0;
  a.unit0 = unit0;
  const int units = n_units;
  if (units < 1) return EBD_OK;
  const int C = ctas_per_unit > 0 ? ctas_per_unit : select_cluster_size(d->n_ctx, units);
  if (C > 1) {
    // a cluster of C CTAs per unit, CTA r holding tokens [r S, (r + 1) S)
    const int per = (d->n_ctx + C - 1) / C;
    const int jg = (per + kGroupTokens - 1) / kGroupTokens;
    const size_t smem = (size_t)jg * kRegThreads * sizeof(float4) + kRegWarps * kHistStride * 4;
    if (cudaFuncSetAttribute(evict_select_smem_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem) != cudaSuccess)
      return EBD_ERR_CUDA;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(units * C));
    cfg.blockDim = dim3(kRegThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)C;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, evict_select_smem_kernel, a, jg) == cudaSuccess)
      return launch_status();
    (void)cudaGetLastError();  // the cluster could not be placed: one CTA per unit below
  }
  const int groups = (d->n_ctx + kGroupTokens - 1) / kGroupTokens;
  if (groups <= kRegMaxGroups) {
    // the limit is set on every launch: with the kernel's static shared memory
    // even 48 KB of dynamic memory is above the default
    const size_t smem = (size_t)groups * kRegThreads * sizeof(float4) + kRegWarps * kHistStride * 4;
    if (cudaFuncSetAttribute(evict_select_smem_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem) != cudaSuccess)
      return EBD_ERR_CUDA;
    evict_select_smem_kernel<<<units, kRegThreads, smem, stream>>>(a, groups);
    return launch_status();
  }
  // certainty bits (padded to 16 bytes), then the per-warp first-digit histograms
  const int words_pad = ((d->n_ctx + 31) / 32 + 3) & ~3;
  const size_t smem = (size_t)words_pad * 4 + (size_t)kSelWarps * 256 * 4;
  if (cudaFuncSetAttribute(evict_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem) != cudaSuccess)
    return EBD_ERR_CUDA;
  evict_select_kernel<<<units, kSelThreads, smem, stream>>>(a, words_pad);
  return launch_status();
}

ebd_status launch_select(const ebd_design* d, const float* scores, const int32_t* n_len,
                         float* pi, uint8_t* mask, int32_t* idx_c, float* logw_c, int32_t* n_kept,
                         int cap, int32_t* dev_status, cudaStream_t stream) {
  return launch_select_range(d, scores, n_len, pi, mask, idx_c, logw_c, n_kept, cap, dev_status,
                             0, d->batch * d->n_kv_heads, stream, 0);
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

ebd_status launch_gather_range(const ebd_design* d, ebd_dtype dtype, const void* K,
                               const void* V, const int32_t* idx_c, const int32_t* n_kept,
                               int cap, void* K_c, void* V_c, int unit0, int n_units,
                               cudaStream_t s) {
  const int eb = dtype == EBD_F32 ? 4 : 2;
  const int cpr = d->head_dim * eb / 16;
  const int units = n_units;
  if (units < 1) return EBD_OK;
  if (units > 65535) return EBD_ERR_UNSUPPORTED;
  const long long items = (long long)cap * cpr;
  long long bx = (items + (long long)kGatherThreads * kGatherUnroll - 1) /
                 ((long long)kGatherThreads * kGatherUnroll);
  if (bx < 1) bx = 1;
  if (bx > 65535) bx = 65535;
  dim3 grid((unsigned)bx, (unsigned)units);
  gather_rows_kernel<<<grid, kGatherThreads, 0, s>>>((const uint4*)K, (const uint4*)V,
                                                     (uint4*)K_c, (uint4*)V_c, idx_c, n_kept,
                                                     d->n_ctx, cap, cpr, unit0);
  return launch_status();
}

ebd_status launch_gather(const ebd_design* d, ebd_dtype dtype, const void* K, const void* V,
                         const int32_t* idx_c, const int32_t* n_kept, int cap, void* K_c,
                         void* V_c, cudaStream_t s) {
  return launch_gather_range(d, dtype, K, V, idx_c, n_kept, cap, K_c, V_c, 0,
                             d->batch * d->n_kv_heads, s);
}

}  // namespace ebd

using namespace ebd;

extern "C" const char* ebd_status_string(ebd_status s) {
  switch (s) {
    case EBD_OK: return "EBD_OK";
    case EBD_ERR_INVALID: return "EBD_ERR_INVALID: invalid argument";
    case EBD_ERR_CAPACITY: return "EBD_ERR_CAPACITY: capacity or workspace too small";
    case EBD_ERR_NONFINITE: return "EBD_ERR_NONFINITE: non-finite input";
    case EBD_ERR_UNSUPPORTED: return "EBD_ERR_UNSUPPORTED: not supported by this build";
    case EBD_ERR_CUDA: return "EBD_ERR_CUDA: CUDA runtime error";
  }
  return "EBD_ERR_UNKNOWN";
}

extern "C" int32_t ebd_abi_version(void) { return 3; }

extern "C" ebd_status ebd_philox_uniforms(uint64_t seed, int32_t layer, int32_t batch,
                                          int32_t n_kv_heads, int32_t n_ctx, uint32_t* x0,
                                          void* stream) {
  if (!x0 || batch < 1 || n_kv_heads < 1 || n_ctx < 1) return EBD_ERR_INVALID;
  const long long total = (long long)batch * n_kv_heads * n_ctx;
  const int threads = 256;
  long long blocks = (total + threads - 1) / threads;
  if (blocks > (long long)sm_count() * 64) blocks = (long long)sm_count() * 64;
  philox_words_kernel<<<(unsigned)blocks, threads, 0, (cudaStream_t)stream>>>(
      seed, layer, n_kv_heads, n_ctx, total, x0);
  return launch_status();
}

extern "C" ebd_status ebd_compute_pi(const ebd_design* design, const float* scores, float* pi,
                                     uint8_t* certain_mask, int32_t* dev_status, void* stream) {
  ebd_status st = check_design(design);
  if (st != EBD_OK) return st;
  if (!scores || !pi) return EBD_ERR_INVALID;
  const float* sc = (const float*)device_address(scores);
  if (!sc) return EBD_ERR_INVALID;
  return launch_select(design, sc, nullptr, pi, certain_mask, nullptr, nullptr, nullptr, 0,
                       dev_status, (cudaStream_t)stream);
}

extern "C" size_t ebd_evict_workspace_bytes(const ebd_design* design, int32_t n_obs) {
  if (!design || n_obs <= 0) return 0;
  const size_t units = (size_t)design->batch * design->n_kv_heads;
  return align_up(units * design->n_ctx * sizeof(float), 256) +
         align_up(units * (size_t)n_obs * sizeof(float), 256);
}

namespace ebd {

// Address under which the kernels read a buffer the caller passed: device or
// managed memory as it is; page-locked host memory through its device mapping
// (the kernels then read it over the host link, only the parts they use);
// nullptr for memory the device cannot address (pageable host memory).
const void* device_address(const void* p) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  switch (at.type) {
    case cudaMemoryTypeDevice:
    case cudaMemoryTypeManaged:
      return p;
    case cudaMemoryTypeHost:
      return at.devicePointer;
    default:
      return nullptr;
  }
}

bool is_device_memory(const void* p) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

// ---- pipelined eviction -------------------------------------------------------
// A select CTA holds a whole SM (1024 threads, the unit's scores in shared
// memory) for tens of microseconds at a low HBM rate, while the row gather is
// HBM-bound and light on the SM.  With more units than SMs the units are cut
// into chunks of one select wave (one unit per SM) and each chunk's
// select -> gather pair runs on its own stream: chunk 0 on the caller's
// stream, the others on side streams forked from it and joined back into it
// by events.  The gather of the first wave then streams while the second wave
// selects, instead of both waves selecting before any row moves.  Chunks
// cover disjoint units, so the outputs do not depend on the schedule.
constexpr int kEvictSideStreams = 3;

struct EvictStreams {
  bool tried = false, ok = false;
  cudaStream_t side[kEvictSideStreams] = {};
  cudaEvent_t fork = nullptr;
  cudaEvent_t join[kEvictSideStreams] = {};
  ~EvictStreams() {
    if (!ok) return;
    for (int i = 0; i < kEvictSideStreams; ++i) {
      cudaStreamDestroy(side[i]);
      cudaEventDestroy(join[i]);
    }
    cudaEventDestroy(fork);
  }
};

// Side streams and events of this host thread on the current device, created
// on first use outside stream capture (nullptr when unavailable: the caller
// then runs the chunks in order on its own stream).
EvictStreams* evict_streams(cudaStream_t s) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    return nullptr;
  }
  static thread_local EvictStreams tl[64];
  EvictStreams& e = tl[dev];
  if (!e.tried) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(s, &cs) != cudaSuccess || cs != cudaStreamCaptureStatusNone) {
      cudaGetLastError();
      return nullptr;  // create nothing while a graph is being captured
    }
    e.tried = true;
    int made = 0;
    bool ok = cudaEventCreateWithFlags(&e.fork, cudaEventDisableTiming) == cudaSuccess;
    for (; ok && made < kEvictSideStreams; ++made) {
      if (cudaStreamCreateWithFlags(&e.side[made], cudaStreamNonBlocking) != cudaSuccess) {
        ok = false;
        break;
      }
      if (cudaEventCreateWithFlags(&e.join[made], cudaEventDisableTiming) != cudaSuccess) {
        cudaStreamDestroy(e.side[made]);
        ok = false;
        break;
      }
    }
    if (!ok) {
      cudaGetLastError();
      for (int i = 0; i < made; ++i) {
        cudaStreamDestroy(e.side[i]);
        cudaEventDestroy(e.join[i]);
      }
      if (e.fork) cudaEventDestroy(e.fork);
    }
    e.ok = ok;
  }
  return e.ok ? &e : nullptr;
}

// E1-E4 for every unit: chunks of one select wave of units, pipelined over streams.
ebd_status select_and_gather(const ebd_design* d, ebd_dtype dtype, const float* scores,
                             const void* K, const void* V, void* K_c, void* V_c, float* logw_c,
                             int32_t* idx_c, int32_t* n_kept, int cap, int32_t* dev_status,
                             cudaStream_t s) {
  const int units = d->batch * d->n_kv_heads;
  // One cluster size for the whole call, so that every chunk splits its units
  // as one launch over all of them would (the float sums of Eq. 2 follow the
  // split).  A chunk is one select wave: an SM per CTA.
  const int C = select_cluster_size(d->n_ctx, units);
  const int chunk = C > 1 ? (sm_count() / C > 0 ? sm_count() / C : 1) : sm_count();
  EvictStreams* es = units > chunk ? evict_streams(s) : nullptr;
  if (!es) {
    ebd_status st = launch_select(d, scores, nullptr, nullptr, nullptr, idx_c, logw_c, n_kept,
                                  cap, dev_status, s);
    if (st != EBD_OK) return st;
    return launch_gather(d, dtype, K, V, idx_c, n_kept, cap, K_c, V_c, s);
  }
  const int n_chunks = (units + chunk - 1) / chunk;
  const int n_side = n_chunks - 1 < kEvictSideStreams ? n_chunks - 1 : kEvictSideStreams;
  if (cudaEventRecord(es->fork, s) != cudaSuccess) return EBD_ERR_CUDA;
  int forked = 0;
  ebd_status st = EBD_OK;
  for (; forked < n_side; ++forked)
    if (cudaStreamWaitEvent(es->side[forked], es->fork, 0) != cudaSuccess) {
      st = EBD_ERR_CUDA;
      break;
    }
  for (int c = 0; st == EBD_OK && c < n_chunks; ++c) {
    const int lane = c % (n_side + 1);
    cudaStream_t cs = lane == 0 ? s : es->side[lane - 1];
    const int u0 = c * chunk;
    const int n = units - u0 < chunk ? units - u0 : chunk;
    st = launch_select_range(d, scores, nullptr, nullptr, nullptr, idx_c, logw_c, n_kept, cap,
                             dev_status, u0, n, cs, C);
    if (st == EBD_OK)
      st = launch_gather_range(d, dtype, K, V, idx_c, n_kept, cap, K_c, V_c, u0, n, cs);
  }
  // every forked stream is joined back, also after an error (a capture needs it)
  for (int i = 0; i < forked; ++i) {
    if (cudaEventRecord(es->join[i], es->side[i]) != cudaSuccess ||
        cudaStreamWaitEvent(s, es->join[i], 0) != cudaSuccess)
      st = EBD_ERR_CUDA;
  }
  return st;
}

}  // namespace ebd

extern "C" ebd_status ebd_evict(const ebd_design* design, ebd_dtype dtype, const void* K,
                                const void* V, const float* scores, const void* q_obs,
                                int32_t n_obs, void* K_c, void* V_c, float* logw_c,
                                int32_t* idx_c, int32_t* n_kept, int32_t capacity,
                                int32_t* dev_status, void* workspace, size_t ws_bytes,
                                void* stream) {
  ebd_status st = check_design(design);
  if (st != EBD_OK) return st;
  if (dtype != EBD_F32 && dtype != EBD_BF16) return EBD_ERR_INVALID;
  if (!K || !V || !K_c || !V_c || !logw_c || !idx_c || !n_kept || !dev_status) return EBD_ERR_INVALID;
  if (capacity < 1) return EBD_ERR_INVALID;
  const int d = design->head_dim;
  const int eb = dtype == EBD_F32 ? 4 : 2;
  if (d < 1 || (d * eb) % 16 != 0) return EBD_ERR_UNSUPPORTED;
  if (!aligned16(K) || !aligned16(V) || !aligned16(K_c) || !aligned16(V_c)) return EBD_ERR_INVALID;
  cudaStream_t s = (cudaStream_t)stream;
  const float* sc = scores;
  if (sc) {  // K, V and the scores may be page-locked host memory
    K = device_address(K);
    V = device_address(V);
    sc = (const float*)device_address(sc);
    if (!K || !V || !sc || !aligned16(K) || !aligned16(V)) return EBD_ERR_INVALID;
  } else {
    // scoring reads every key: K and the observation queries in device memory
    if (!q_obs || n_obs < 1) return EBD_ERR_INVALID;
    if (!is_device_memory(K) || !is_device_memory(q_obs)) return EBD_ERR_UNSUPPORTED;
    V = device_address(V);
    if (!V) return EBD_ERR_INVALID;
    const size_t need = ebd_evict_workspace_bytes(design, n_obs);
    if (!workspace || ws_bytes < need) return EBD_ERR_CAPACITY;
    const size_t units = (size_t)design->batch * design->n_kv_heads;
    float* ws_scores = (float*)workspace;
    float* ws_lse = (float*)((char*)workspace + align_up(units * design->n_ctx * sizeof(float), 256));
    st = launch_score(dtype, design->batch, design->n_kv_heads, d, design->n_ctx, n_obs, q_obs, K,
                      ws_scores, ws_lse, dev_status, s);
    if (st != EBD_OK) return st;
    sc = ws_scores;
  }
  return select_and_gather(design, dtype, sc, K, V, K_c, V_c, logw_c, idx_c, n_kept, capacity,
                           dev_status, s);
}

extern "C" ebd_status ebd_select(const ebd_design* design, const float* scores, int32_t* idx_c,
                                 float* logw_c, int32_t* n_kept, int32_t capacity,
                                 int32_t* dev_status, void* stream) {
  ebd_status st = check_design(design);
  if (st != EBD_OK) return st;
  if (!scores || !idx_c || !logw_c || !n_kept || !dev_status || capacity < 1) return EBD_ERR_INVALID;
  const float* sc = (const float*)device_address(scores);
  if (!sc) return EBD_ERR_INVALID;
  return launch_select(design, sc, nullptr, nullptr, nullptr, idx_c, logw_c, n_kept, capacity,
                       dev_status, (cudaStream_t)stream);
}

extern "C" ebd_status ebd_gather(const ebd_design* design, ebd_dtype dtype, const void* K,
                                 const void* V, const int32_t* idx_c, const int32_t* n_kept,
                                 int32_t capacity, void* K_c, void* V_c, void* stream) {
  ebd_status st = check_design(design);
  if (st != EBD_OK) return st;
  if (dtype != EBD_F32 && dtype != EBD_BF16) return EBD_ERR_INVALID;
  if (!K || !V || !idx_c || !n_kept || !K_c || !V_c || capacity < 1) return EBD_ERR_INVALID;
  const int eb = dtype == EBD_F32 ? 4 : 2;
  if (design->head_dim < 1 || (design->head_dim * eb) % 16 != 0) return EBD_ERR_UNSUPPORTED;
  if (!aligned16(K) || !aligned16(V) || !aligned16(K_c) || !aligned16(V_c)) return EBD_ERR_INVALID;
  K = device_address(K);  // page-locked host rows are read over the host link
  V = device_address(V);
  if (!K || !V || !aligned16(K) || !aligned16(V)) return EBD_ERR_INVALID;
  return launch_gather(design, dtype, K, V, idx_c, n_kept, capacity, K_c, V_c,
                       (cudaStream_t)stream);
}
