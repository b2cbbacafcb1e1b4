// The per-tile step of the tensor-core certified decode (bf16 compact cache,
// head_dim 64/128, G <= 8), shared by the persistent split-K kernel
// (decode_mma.cu) and the cluster kernel (decode_cluster.cu).
//
// One warp, one 16-token tile of one unit (Eq. 3, Theorem 2, Eq. 4):
//   S[16 x 16]  = Qpad[16 x d] . K_tile^T       (rows 0..G-1 = query heads,
//                                                rows 8..15 = 0; 2 x d/16 mma)
//   w = 2^(S log2e/sqrt(d) + log2e log(1/pi) - M), u = (1 - pi) w^2
//   P[16 x 16]  = [w (rows 0..7); u (rows 8..15)] as bf16 hi + bf16 lo parts
//   acc[16 x d] += P_hi . V_tile + P_lo . V_tile   (rows 0..7: o, rows 8..15: A1)
// plus l = sum w, U = sum u, A2 = sum u ||v - c||^2 and the range-bound
// maxima cmax = max sqrt(u) ||v - c||, umax = max sqrt(u).  c is the unit's
// centring row (centre_row in decode.cuh), so that the second moment does not
// carry the values' common mean: the combine forms
// V_hat l^2 = A2 - 2 (y - c).(A1 - U c) + ||y - c||^2 U, every term of the
// size of the spread of v around y, and the one-pass range bound
// (cmax + ||y - c|| umax) / l.  The hi/lo split keeps ~16 mantissa bits of the
// weights on bf16 tensor cores; ||v - c||^2 per token comes from the same V
// fragments.  The running maximum M is updated lazily:
// accumulators are rescaled only when a row's maximum grows by more than 2^8,
// so weights stay below 2^8 and u below 2^16.
//
// Groups of at most four query heads (PACK) use the MMA rows the heads leave
// free: query rows 4..7 repeat rows 0..3, so lanes 16..31 compute the same
// weights bit for bit, and the [w; u] V product takes the hi parts of head g
// in rows g and g + 8 and the lo parts in rows g + 4 and g + 12 -- one MMA per
// 8 columns instead of two.  o and A1 are then the sums of rows g and g + 4
// (resp. g + 8 and g + 12), added when the state is stored.
//
// A tile stage holds K and V as 64-column (128-byte) halves of 16 rows in the
// 128-byte swizzle pattern (chunk ch of row r at r * 128 + ((ch ^ (r & 7)) << 4))
// that ldmatrix reads without bank conflicts, then V, and 16 floats of
// log(1/pi) in a separate array.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

#include <type_traits>

#include "common.cuh"
#include "decode.cuh"
#include "ptx.cuh"

namespace ebd {

constexpr int kMmaTile = 16;
constexpr int kMmaConsumers = 8;  // warps per CTA
constexpr int kMmaThreads = kMmaConsumers * 32;
constexpr float kRescaleLog2 = 8.f;

// Programmatic dependent launch: a kernel launched with programmatic stream
// serialization may start while its predecessor in the stream runs; it must
// wait before reading the predecessor's outputs or writing anything.  A
// kernel lets its own dependents launch early with launch_dependents.
__device__ __forceinline__ void grid_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void grid_dependency_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

template <int D>
struct MmaTileLayout {
  static constexpr int kHalves = D / 64;             // 64-column (128-byte) boxes per row
  static constexpr int kBoxBytes = kMmaTile * 128;   // one box: 16 rows x 128 B
  static constexpr int kStageBytes = 2 * kHalves * kBoxBytes;
};

// A warp's running state over tiles of one unit, per lane: acc rows 0..7 are
// o of query heads 0..7, rows 8..15 are A1; qa the query fragments.
template <int D>
struct TileAcc {
  float acc[D / 8][4];
  float M2, l, U, A2, cmax, umax;  // M2: running maximum in log2 units
  uint32_t qa[D / 16][2];
  // -c as bf16 pairs: channel 16 jp + lane/4 (low half), 16 jp + 8 + lane/4
  // (high half) -- the channels of this lane's V fragments
  uint32_t cneg[D / 16];
};

// Start a unit: its G query rows (row u * qstride + g of Q) as mma A fragments
// (rows >= G are zero; with PACK, rows 4..7 repeat rows 0..3), its centring
// row (Vc: the compact V cache, cap rows per unit; n_u: the unit's retained
// rows), and empty sums.
template <int D, bool PACK>
__device__ __forceinline__ void tile_acc_begin(TileAcc<D>& t, const __nv_bfloat16* Q,
                                               const __nv_bfloat16* Vc, int u, int G, int qstride,
                                               int cap, int n_u, int lane) {
  const int q = lane & 3;
  {
    // channels of this lane's V fragments: 16 jp + lane/4 and 16 jp + 8 + lane/4
    const int col = lane >> 2;
    const int cr = centre_row(n_u);
    const unsigned short* crow =
        reinterpret_cast<const unsigned short*>(Vc + ((size_t)u * cap + (cr < 0 ? 0 : cr)) * D);
#pragma unroll
    for (int jp = 0; jp < D / 16; ++jp) {
      const uint32_t lo = cr < 0 ? 0u : __ldg(crow + 16 * jp + col);
      const uint32_t hi = cr < 0 ? 0u : __ldg(crow + 16 * jp + 8 + col);
      t.cneg[jp] = (lo | (hi << 16)) ^ 0x80008000u;  // both halves negated
    }
  }
  const int g = PACK ? (lane >> 2) & 3 : lane >> 2;  // query row of this lane's A fragments
  const uint32_t* qrow =
      reinterpret_cast<const uint32_t*>(Q + ((size_t)u * qstride + (g < G ? g : 0)) * D);
#pragma unroll
  for (int kk = 0; kk < D / 16; ++kk) {
    t.qa[kk][0] = g < G ? __ldg(qrow + 8 * kk + q) : 0u;
    t.qa[kk][1] = g < G ? __ldg(qrow + 8 * kk + 4 + q) : 0u;
  }
#pragma unroll
  for (int j = 0; j < D / 8; ++j) t.acc[j][0] = t.acc[j][1] = t.acc[j][2] = t.acc[j][3] = 0.f;
  t.M2 = -INFINITY;
  t.l = t.U = t.A2 = t.cmax = t.umax = 0.f;
}

// cp.async copies of one tile (rows row0 .. row0 + 15 of the compact cache)
// into a stage: every lane copies 16-byte chunks of K and V, lanes 0-3 the
// tile's log(1/pi).  The caller commits the group.
template <int D>
__device__ __forceinline__ void tile_copy(unsigned char* st, float* lw_dst,
                                          const __nv_bfloat16* __restrict__ Kc,
                                          const __nv_bfloat16* __restrict__ Vc,
                                          const float* __restrict__ logw, size_t row0, int lane) {
  using L = MmaTileLayout<D>;
  constexpr int CPR = D / 8;                // 16-byte chunks per row
  constexpr int PER = kMmaTile * CPR / 32;  // chunks per lane per tile (K or V)
#pragma unroll
  for (int i = 0; i < PER; ++i) {
    const int c = lane + 32 * i;
    const int r = c / CPR, ch = c - r * CPR;
    const int off = (ch >> 3) * L::kBoxBytes + r * 128 + (((ch & 7) ^ (r & 7)) << 4);
    const size_t src = (row0 + r) * D + ch * 8;
    cp_async16(st + off, Kc + src);
    cp_async16(st + L::kHalves * L::kBoxBytes + off, Vc + src);
  }
  if (lane < kMmaTile / 4) cp_async16(lw_dst + 4 * lane, logw + row0 + 4 * lane);
}

// Fold one tile (stage at shared address kbase, its log(1/pi) at lw; tokens
// >= n_valid are outside the unit) into the warp's state.
template <int D, bool PACK>
__device__ __forceinline__ void tile_consume(TileAcc<D>& t, uint32_t kbase, const float* lw,
                                             int n_valid, int lane, float kscale) {
  using L = MmaTileLayout<D>;
  const int q = lane & 3;
  const uint32_t vbase = kbase + L::kHalves * L::kBoxBytes;

  // ---- S = Q K^T ---------------------------------------------------------
  // even and odd k-steps accumulate separately: two dependent MMA chains of
  // D/32 per 8 tokens instead of one of D/16
  float sc0[4] = {0.f, 0.f, 0.f, 0.f}, sc1[4] = {0.f, 0.f, 0.f, 0.f};
  {
    float sd0[4] = {0.f, 0.f, 0.f, 0.f}, sd1[4] = {0.f, 0.f, 0.f, 0.f};
    const int tok = ((lane >> 4) << 3) + (lane & 7);
    const int half_sel = (lane >> 3) & 1;
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      const int chunk = 2 * kk + half_sel;
      const uint32_t addr =
          kbase + (chunk >> 3) * L::kBoxBytes + tok * 128 + (((chunk & 7) ^ (tok & 7)) << 4);
      uint32_t b0, b1, b2, b3;
      ldsm_x4(addr, b0, b1, b2, b3);
      mma_bf16_16816(kk & 1 ? sd0 : sc0, t.qa[kk][0], 0u, t.qa[kk][1], 0u, b0, b1);
      mma_bf16_16816(kk & 1 ? sd1 : sc1, t.qa[kk][0], 0u, t.qa[kk][1], 0u, b2, b3);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      sc0[i] += sd0[i];
      sc1[i] += sd1[i];
    }
  }

  // ---- weights -----------------------------------------------------------
  const float2 lwa = *reinterpret_cast<const float2*>(lw + 2 * q);
  const float2 lwb = *reinterpret_cast<const float2*>(lw + 8 + 2 * q);
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
  if (mx > t.M2 + kRescaleLog2) {
    const float f = exp2f(t.M2 - mx), f2 = f * f;
#pragma unroll
    for (int jj = 0; jj < D / 8; ++jj) {
      t.acc[jj][0] *= f;
      t.acc[jj][1] *= f;
      t.acc[jj][2] *= f2;
      t.acc[jj][3] *= f2;
    }
    t.l *= f;
    t.U *= f2;
    t.A2 *= f2;
    t.cmax *= f;
    t.umax *= f;
    t.M2 = mx;
  }
  // 1 - pi and its square root depend on the token only: lane L computes
  // them for token L % 16 (0 past the unit) and the lanes that use them read
  // them with shuffles
  float omp_t, som_t;
  {
    const int tt = lane & (kMmaTile - 1);
    omp_t = tt < n_valid ? one_minus_exp_neg(lw[tt]) : 0.f;
    som_t = sqrtf(omp_t);
  }
  float wv[4], uv[4], suv[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    wv[i] = exp2f(x[i] - t.M2);
    const float omp = __shfl_sync(0xffffffffu, omp_t, tk[i]);  // 1 - pi
    uv[i] = omp * wv[i] * wv[i];
    suv[i] = __shfl_sync(0xffffffffu, som_t, tk[i]) * wv[i];
    t.umax = fmaxf(t.umax, suv[i]);
  }
  const uint32_t h0 = pack_bf16(wv[0], wv[1]), h1 = pack_bf16(uv[0], uv[1]);
  const uint32_t h2 = pack_bf16(wv[2], wv[3]), h3 = pack_bf16(uv[2], uv[3]);
  const uint32_t r0 = pack_bf16(wv[0] - bf16_lo(h0), wv[1] - bf16_hi(h0));
  const uint32_t r1 = pack_bf16(uv[0] - bf16_lo(h1), uv[1] - bf16_hi(h1));
  const uint32_t r2 = pack_bf16(wv[2] - bf16_lo(h2), wv[3] - bf16_hi(h2));
  const uint32_t r3 = pack_bf16(uv[2] - bf16_lo(h3), uv[3] - bf16_hi(h3));
  // The scalar sums use exactly the weights the tensor cores multiply with
  // (hi + lo), so that V_hat = (A2 - 2 (y - c).(A1 - U c) + |y - c|^2 U) / l^2
  // stays consistent when few tail rows carry it.
  const float wt[4] = {bf16_lo(h0) + bf16_lo(r0), bf16_hi(h0) + bf16_hi(r0),
                       bf16_lo(h2) + bf16_lo(r2), bf16_hi(h2) + bf16_hi(r2)};
  const float ut[4] = {bf16_lo(h1) + bf16_lo(r1), bf16_hi(h1) + bf16_hi(r1),
                       bf16_lo(h3) + bf16_lo(r3), bf16_hi(h3) + bf16_hi(r3)};
  t.l += (wt[0] + wt[1]) + (wt[2] + wt[3]);
  t.U += (ut[0] + ut[1]) + (ut[2] + ut[3]);
  // PACK: lanes 0..15 feed the hi parts (rows g, g + 8), lanes 16..31 the lo
  // parts of the same head (rows g + 4, g + 12)
  const bool upper = PACK && lane >= 16;
  const uint32_t p0 = upper ? r0 : h0, p1 = upper ? r1 : h1;
  const uint32_t p2 = upper ? r2 : h2, p3 = upper ? r3 : h3;

  // ---- acc += P V, ||v - c||^2 ----------------------------------------------
  // Rows past the unit (the last tile only) are zeroed before use: the buffer
  // may hold anything there, and 0 * NaN would reach the sums.
  float2 vc01 = make_float2(0.f, 0.f), vc23 = make_float2(0.f, 0.f);
  auto pv_pass = [&](auto masked) {
    constexpr bool kMasked = decltype(masked)::value;
    const uint32_t m01 =
        (tk[0] < n_valid ? 0x0000ffffu : 0u) | (tk[1] < n_valid ? 0xffff0000u : 0u);
    const uint32_t m23 =
        (tk[2] < n_valid ? 0x0000ffffu : 0u) | (tk[3] < n_valid ? 0xffff0000u : 0u);
    const int tok = ((lane >> 3) & 1) * 8 + (lane & 7);
    const int chunk_sel = lane >> 4;
#pragma unroll
    for (int jp = 0; jp < D / 16; ++jp) {
      const int chunk = 2 * jp + chunk_sel;
      const uint32_t addr =
          vbase + (chunk >> 3) * L::kBoxBytes + tok * 128 + (((chunk & 7) ^ (tok & 7)) << 4);
      uint32_t v0, v1, v2, v3;
      ldsm_x4_trans(addr, v0, v1, v2, v3);
      if constexpr (kMasked) {
        v0 &= m01;
        v2 &= m01;
        v1 &= m23;
        v3 &= m23;
      }
      const float2 f0 = make_float2(bf16_lo(v0), bf16_hi(v0));
      const float2 f1 = make_float2(bf16_lo(v1), bf16_hi(v1));
      const float2 f2 = make_float2(bf16_lo(v2), bf16_hi(v2));
      const float2 f3 = make_float2(bf16_lo(v3), bf16_hi(v3));
      // v - c: exact for bf16 v and c of similar magnitude (masked rows give
      // -c, finite, and carry u = 0)
      const float cl = bf16_lo(t.cneg[jp]), ch = bf16_hi(t.cneg[jp]);
      const float2 e0 = __fadd2_rn(f0, make_float2(cl, cl));
      const float2 e1 = __fadd2_rn(f1, make_float2(cl, cl));
      const float2 e2 = __fadd2_rn(f2, make_float2(ch, ch));
      const float2 e3 = __fadd2_rn(f3, make_float2(ch, ch));
      vc01 = __ffma2_rn(e0, e0, __ffma2_rn(e2, e2, vc01));
      vc23 = __ffma2_rn(e1, e1, __ffma2_rn(e3, e3, vc23));
      if constexpr (PACK) {
        mma_bf16_16816(t.acc[2 * jp], p0, p1, p2, p3, v0, v1);
        mma_bf16_16816(t.acc[2 * jp + 1], p0, p1, p2, p3, v2, v3);
      } else {
        mma_bf16_16816(t.acc[2 * jp], h0, h1, h2, h3, v0, v1);
        mma_bf16_16816(t.acc[2 * jp], r0, r1, r2, r3, v0, v1);
        mma_bf16_16816(t.acc[2 * jp + 1], h0, h1, h2, h3, v2, v3);
        mma_bf16_16816(t.acc[2 * jp + 1], r0, r1, r2, r3, v2, v3);
      }
    }
  };
  if (n_valid >= kMmaTile) pv_pass(std::false_type{});
  else pv_pass(std::true_type{});
  // every lane's reads of this stage are done before it is refilled
  __syncwarp();
  float vc[4] = {vc01.x, vc01.y, vc23.x, vc23.y};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    vc[i] += __shfl_xor_sync(0xffffffffu, vc[i], 4);
    vc[i] += __shfl_xor_sync(0xffffffffu, vc[i], 8);
    vc[i] += __shfl_xor_sync(0xffffffffu, vc[i], 16);
    t.A2 = fmaf(ut[i], vc[i], t.A2);
    t.cmax = fmaxf(t.cmax, suv[i] * sqrtf(vc[i]));
  }
}

// Write the warp's state as partial records: head g = lane / 4 (g < G) at
// rec + g * rec_floats(D): [M (natural log), l, U, A2 (about the unit's
// centring row), cmax, umax, -, -, o[D], A1[D]].  The scalar sums are first completed over the four lanes of
// a head.
template <int D, bool PACK>
__device__ __forceinline__ void tile_acc_store(TileAcc<D>& t, float* rec_base, int G, int lane) {
  constexpr int REC = rec_floats(D);
  const int g = lane >> 2, q = lane & 3;
  if constexpr (PACK) {  // add the lo rows (lanes 16..31) to the hi rows
#pragma unroll
    for (int j = 0; j < D / 8; ++j)
#pragma unroll
      for (int k = 0; k < 4; ++k) t.acc[j][k] += __shfl_xor_sync(0xffffffffu, t.acc[j][k], 16);
  }
#pragma unroll
  for (int o = 1; o <= 2; o <<= 1) {
    t.l += __shfl_xor_sync(0xffffffffu, t.l, o);
    t.U += __shfl_xor_sync(0xffffffffu, t.U, o);
    t.A2 += __shfl_xor_sync(0xffffffffu, t.A2, o);
    t.cmax = fmaxf(t.cmax, __shfl_xor_sync(0xffffffffu, t.cmax, o));
    t.umax = fmaxf(t.umax, __shfl_xor_sync(0xffffffffu, t.umax, o));
  }
  if (g < G) {
    float* rec = rec_base + (size_t)g * REC;
    if (q == 0) {
      rec[kRecM] = t.M2 == -INFINITY ? -INFINITY : t.M2 * kLn2;
      rec[kRecL] = t.l;
      rec[kRecU] = t.U;
      rec[kRecA2] = t.A2;
      rec[kRecCmax] = t.cmax;
      rec[kRecUmax] = t.umax;
    }
#pragma unroll
    for (int j = 0; j < D / 8; ++j) {
      *reinterpret_cast<float2*>(rec + kRecHead + 8 * j + 2 * q) =
          make_float2(t.acc[j][0], t.acc[j][1]);
      *reinterpret_cast<float2*>(rec + kRecHead + D + 8 * j + 2 * q) =
          make_float2(t.acc[j][2], t.acc[j][3]);
    }
  }
}

}  // namespace ebd
