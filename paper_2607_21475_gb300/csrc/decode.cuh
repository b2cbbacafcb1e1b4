// Split-K record layout and launch plumbing shared by the certified-decode kernels.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/ebd.h"
#include "common.cuh"

namespace ebd {

// Centring row of a unit with n retained rows: the middle one, or -1 (c = 0)
// for an empty unit.  Every partial record of a unit takes its second moment
// A2 = sum u ||v - c||^2 about the same row c = V_c[centre_row(n)], and the
// combine finishes
//   V_hat l^2 = sum u ||v - y||^2 = A2 - 2 (y - c).(A1 - U c) + ||y - c||^2 U,
// so no term carries the values' common mean (with A2 about the origin, a mean
// of 16 on every channel makes each term ~256 times V_hat l^2 and float32
// rounding of the sums shows in V_hat).  Any retained row serves: c only has
// to lie within the spread of the values.  The one-pass range bound of Eq. 4
// is taken about the same row: (max sqrt(u) ||v - c|| + ||y - c|| max sqrt(u)) / l.
__host__ __device__ constexpr int centre_row(int n) { return n > 0 ? (n - 1) / 2 : -1; }

// Columns PER * lane .. + PER - 1 of the centring row of a unit (n retained
// rows, cap rows per unit in Vc), as floats; zeros for an empty unit.
template <typename T, int D, int PER>
__device__ __forceinline__ void load_centre(const T* Vc, long long unit, int cap, int n, int lane,
                                            float (&c)[PER]) {
  const int cr = centre_row(n);
  const T* row = Vc + ((size_t)unit * cap + (cr < 0 ? 0 : cr)) * D + PER * lane;
#pragma unroll
  for (int e = 0; e < PER; ++e) c[e] = cr < 0 ? 0.f : to_f32(row[e]);
}

// Finish one query head from its combined sums (Eq. 3, Theorem 2): y_hat =
// o / l on this lane's PER columns, ||y_hat||, ||y_hat - c|| and
//   V_hat = (A2 - 2 (y - c).(A1 - U c) + ||y - c||^2 U) / l^2
// with A2 taken about the centring row c (every lane gets the warp's sums).
template <int PER>
__device__ __forceinline__ void finish_head(const float (&o)[PER], const float (&a1)[PER],
                                            const float (&c)[PER], float l, float U, float A2,
                                            float (&yv)[PER], float& ynorm, float& ycnorm,
                                            float& var) {
  float yy = 0.f, ycyc = 0.f, yca = 0.f;
#pragma unroll
  for (int e = 0; e < PER; ++e) {
    yv[e] = o[e] / l;
    yy = fmaf(yv[e], yv[e], yy);
    const float yc = yv[e] - c[e];
    const float a1c = fmaf(-U, c[e], a1[e]);
    ycyc = fmaf(yc, yc, ycyc);
    yca = fmaf(yc, a1c, yca);
  }
  yy = warp_sum(yy);
  ycyc = warp_sum(ycyc);
  yca = warp_sum(yca);
  ynorm = sqrtf(yy);
  ycnorm = sqrtf(ycyc);
  var = fmaxf(0.f, (A2 - 2.f * yca + ycyc * U) / (l * l));
}

// One partial record per (unit, split slot, query head of the group), floats:
//   [M, l, U, A2, cmax, umax, pad, pad, o[0..D), A1[0..D)]
// (16-byte multiple, so o and A1 can be read as float4).  w-terms (l, o,
// cmax, umax) scale by e^(M_old - M_new) on a merge, u-terms (U, A2, A1) by
// its square.  An empty record has M = -inf and zeros.
enum : int { kRecM = 0, kRecL = 1, kRecU = 2, kRecA2 = 3, kRecCmax = 4, kRecUmax = 5, kRecHead = 8 };

__host__ __device__ constexpr int rec_floats(int D) { return kRecHead + 2 * D; }
__host__ __device__ constexpr bool rec_is_squared(int e, int D) {
  return e == kRecU || e == kRecA2 || e >= kRecHead + D;
}

// Groups of more than 8 query heads are decoded in slices of at most 8 heads
// (one pass over the compact cache each): `group` is the slice's head count,
// `gstride` the group size of the Q / output layout (query head g of unit u
// of the slice at row u * gstride + g of the slice's Q and output pointers,
// which the host offsets to the slice's first head).
struct DecodeArgs {
  const void* Q;          // [B, Hkv*G, D]
  const void* Kc;         // [units, cap, D]
  const void* Vc;         // [units, cap, D]
  const float* logw;      // [units, cap]
  const int32_t* n_kept;  // [units]
  int cap;
  int n_kv_heads;
  int group;
  int gstride;
  int splits;             // split slots per unit in `part`
  int tokens_per_split;   // CUDA-core path: token range of one split
  float* part;            // [units, splits, G, rec_floats(D)]
  float* y;               // exact range pass: final y_hat (read)
  float* lse;             // exact range pass: final lse (read)
  float* b_t;             // exact range pass: running max (atomicMax)
  int32_t* dev_status;
};

struct ReduceArgs {
  const float* part;         // CUDA-core path: [units, splits, G, rec_floats(D)]
  const void* Vc;            // [units, cap, D]: the centring rows (CUDA-core path)
  const int32_t* n_kept;     // [units]
  int cap;
  int splits;                // records per unit
  int group;
  int gstride;
  float* y;
  float* lse;
  float* var;
  float* b_t;
  float* radius;
  float log_inv_delta;
  float eps0;
  bool exact;
};

struct DecodePlan {
  bool fast = false;         // the tensor-core path applies to this request
  int splits = 1;            // CUDA-core path: splits per unit
  int tokens_per_split = 0;  // CUDA-core path
  int ctas = 0;              // tensor-core path: persistent grid size
  size_t ws_bytes = 0;       // the larger of the two paths' needs
};

DecodePlan plan_decode(ebd_dtype dtype, int batch, int n_kv_heads, int group, int head_dim,
                       int capacity);

// Argument checks of ebd_certified_decode (everything but the workspace), so
// that its variants answer a bad request with the same status.
ebd_status check_decode_args(ebd_dtype dtype, int32_t batch, int32_t n_kv_heads, int32_t group,
                             int32_t head_dim, const void* Q, const void* K_c, const void* V_c,
                             const float* logw_c, const int32_t* n_kept, int32_t capacity,
                             float delta, float eps0, ebd_range_mode range_mode, const float* y,
                             const float* lse, const float* var_hat, const float* b_t,
                             const float* radius);

// Tensor-core path (decode_mma.cu): decode kernel, then a merge kernel
// launched as its programmatic dependent (plus a prefix kernel above 4096
// units).  `ws`: the workspace.
bool fast_decode_supported(ebd_dtype dtype, int group, int head_dim, int capacity);
bool fast_decode_usable(const DecodeArgs& a, const ReduceArgs& r, int units);
void fast_decode_plan(DecodePlan& p, long long units, int group, int head_dim);
ebd_status launch_fast_decode(ebd_dtype dtype, int head_dim, const DecodePlan& plan,
                              const DecodeArgs& a, const ReduceArgs& r, int units, void* ws,
                              cudaStream_t stream);

// Cluster path (decode_cluster.cu): CTAs per unit (0 when the path does not
// apply), and the launch (same arguments as the tensor-core path; no
// workspace).
int cluster_decode_size(int units, int cap);
ebd_status launch_cluster_decode(int head_dim, const DecodeArgs& d, const ReduceArgs& r,
                                 int units, cudaStream_t stream);

}  // namespace ebd
