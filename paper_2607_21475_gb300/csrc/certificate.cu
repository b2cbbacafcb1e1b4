// Deployed certificate of a sequence (the experimental setup of Section 5 and
// its appendix): at each of the first six decode steps the radii r_t of
// Eq. (4), at delta = 0.1, of every fourth query head of every layer are
// averaged; the certificate is the maximum of these step averages, and the
// label-free red-flag rule raises a sequence whose certificate reaches
// tau = 1.  One warp per batch row adds its L * ceil(Hq / stride) radii in a
// fixed order (lane-strided terms, then a fixed shuffle tree), so the result
// does not depend on scheduling.
#include <cuda_runtime.h>

#include "common.cuh"
#include "internal.h"

namespace ebd {

constexpr int kCertWarps = 4;

__global__ void __launch_bounds__(kCertWarps * 32)
    certificate_update_kernel(const float* __restrict__ radius, int n_layers, int batch,
                              int n_q_heads, int head_stride, float tau, int first_step,
                              float* __restrict__ step_mean, float* __restrict__ cert,
                              int32_t* __restrict__ red_flag) {
  const int b = blockIdx.x * kCertWarps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (b >= batch) return;
  const int nh = (n_q_heads + head_stride - 1) / head_stride;  // heads 0, stride, 2 stride, ...
  const long long terms = (long long)n_layers * nh;
  float s = 0.f;
  for (long long k = lane; k < terms; k += 32) {
    const int l = (int)(k / nh), h = (int)(k - (long long)l * nh) * head_stride;
    s += radius[((size_t)l * batch + b) * n_q_heads + h];
  }
  s = warp_sum(s);
  if (lane == 0) {
    const float mean = s / (float)terms;
    const float c = first_step ? mean : fmaxf(cert[b], mean);
    cert[b] = c;
    if (step_mean) step_mean[b] = mean;
    if (red_flag) red_flag[b] = c >= tau ? 1 : 0;
  }
}

}  // namespace ebd

using namespace ebd;

extern "C" ebd_status ebd_certificate_update(const float* radius, int32_t n_layers, int32_t batch,
                                             int32_t n_q_heads, int32_t head_stride, float tau,
                                             int32_t first_step, float* step_mean, float* cert,
                                             int32_t* red_flag, void* stream) {
  if (!radius || !cert || n_layers < 1 || batch < 1 || n_q_heads < 1 || head_stride < 1)
    return EBD_ERR_INVALID;
  if ((long long)n_layers * batch * n_q_heads > 0x7fffffffLL) return EBD_ERR_UNSUPPORTED;
  const int blocks = (batch + kCertWarps - 1) / kCertWarps;
  certificate_update_kernel<<<blocks, kCertWarps * 32, 0, (cudaStream_t)stream>>>(
      radius, n_layers, batch, n_q_heads, head_stride, tau, first_step ? 1 : 0, step_mean, cert,
      red_flag);
  return launch_status();
}
