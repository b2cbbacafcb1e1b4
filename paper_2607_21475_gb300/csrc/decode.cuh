// Split-K record layout and launch plumbing shared by the certified-decode kernels.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/ebd.h"

namespace ebd {

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

struct DecodeArgs {
  const void* Q;          // [B, Hkv*G, D]
  const void* Kc;         // [units, cap, D]
  const void* Vc;         // [units, cap, D]
  const float* logw;      // [units, cap]
  const int32_t* n_kept;  // [units]
  int cap;
  int n_kv_heads;
  int group;
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
  int splits;                // records per unit
  int group;
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
