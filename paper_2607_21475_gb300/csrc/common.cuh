// Device-side helpers shared by the EBD kernels (GB300, sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/ebd.h"

namespace ebd {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// ---------------------------------------------------------------------------
// Element access for the two storage types of K, V and queries.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }

// ---------------------------------------------------------------------------
// Warp / block reductions.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ int warp_sum(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_min(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds of two 32x32
// multiplications whose high halves are XORed with the remaining counter
// words and the key; the key takes a Weyl step between rounds.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint2 k) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k.x += 0x9E3779B9u;
      k.y += 0xBB67AE85u;
    }
    const uint32_t hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo0 = 0xD2511F53u * c.x;
    const uint32_t hi1 = __umulhi(0xCD9E8D57u, c.z);
    const uint32_t lo1 = 0xCD9E8D57u * c.z;
    c = make_uint4(hi1 ^ c.y ^ k.x, lo1, hi0 ^ c.w ^ k.y, lo0);
  }
  return c;
}

// The four Philox words for tokens 4q .. 4q+3 of unit (b, kvh) in `layer`:
// counter (q, kv head, layer, batch row), key (seed low, seed high).
__device__ __forceinline__ uint4 draw_block(uint64_t seed, int layer, int b, int kvh, int q) {
  const uint4 ctr = make_uint4((uint32_t)q, (uint32_t)kvh, (uint32_t)layer, (uint32_t)b);
  const uint2 key = make_uint2((uint32_t)(seed & 0xffffffffu), (uint32_t)(seed >> 32));
  return philox4x32_10(ctr, key);
}

__device__ __forceinline__ uint32_t word_of(const uint4& w, int r) {
  return r == 0 ? w.x : (r == 1 ? w.y : (r == 2 ? w.z : w.w));
}

// Philox word of token i: word i % 4 of the call for tokens 4(i/4) .. 4(i/4)+3.
__device__ __forceinline__ uint32_t draw_word(uint64_t seed, int layer, int b, int kvh, int i) {
  return word_of(draw_block(seed, layer, b, kvh, i >> 2), i & 3);
}

// Uniform in [0,1) from the top 24 bits of a Philox word; exact in float32.
__device__ __forceinline__ float word_to_uniform(uint32_t x0) {
  return (float)(x0 >> 8) * 5.9604644775390625e-08f;  // 2^-24
}

// Order-preserving map float -> uint32 (larger float -> larger key);
// -0.0 is folded onto +0.0 first so equal floats give equal keys.
__device__ __forceinline__ uint32_t orderable_key(float s) {
  s = s + 0.0f;
  const uint32_t b = __float_as_uint(s);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// 1 - e^-x for x >= 0 (x = log(1/pi), so the result is 1 - pi).  Below 0.25
// the Taylor series to x^6 (truncation < 5e-8 relative) avoids the
// cancellation of 1 - e^-x; above it, 1 - e^-x >= 0.22 and exp2 suffices.
__device__ __forceinline__ float one_minus_exp_neg(float x) {
  if (x < 0.25f) {
    return x * (1.f - x * (0.5f - x * (1.f / 6.f - x * (1.f / 24.f - x * (1.f / 120.f - x * (1.f / 720.f))))));
  }
  return 1.f - exp2f(-x * kLog2e);
}

__device__ __forceinline__ void raise_status(int32_t* st, int32_t bits) {
  if (st) atomicOr(st, bits);
}

}  // namespace ebd
