// Host-side declarations shared by the translation units of libebd.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/ebd.h"

namespace ebd {

inline ebd_status cuda_status(cudaError_t e) { return e == cudaSuccess ? EBD_OK : EBD_ERR_CUDA; }

// Last launch error of this thread, mapped to a status (clears the error).
inline ebd_status launch_status() { return cuda_status(cudaGetLastError()); }

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Number of SMs of the current device (cached per device).
int sm_count();

// E0: accumulated attention scores into `scores` using `workspace` for the
// per-row log-sum-exp.  Arguments validated by the caller; dev_status nullable.
ebd_status launch_score(ebd_dtype dtype, int batch, int n_kv_heads, int head_dim, int n_ctx,
                        int n_obs, const void* q_obs, const void* K, float* scores,
                        float* lse_ws, int32_t* dev_status, cudaStream_t stream);

// E0 on tcgen05 with tensor-memory accumulators (score_tc.cu): bf16,
// head_dim 64/128, at most 512 observation rows, 16-byte aligned inputs.
bool score_tc_supported(ebd_dtype dtype, int head_dim, int n_obs, const void* q_obs,
                        const void* K);
ebd_status launch_score_tc(int units, int head_dim, int n_ctx, int n_obs, const void* q_obs,
                           const void* K, float* scores, float* lse, int32_t* dev_status,
                           cudaStream_t s);

// E0 on mma.sync (score_mma.cu): bf16, head_dim 64/128, 16-byte aligned inputs.
bool score_mma_supported(ebd_dtype dtype, int head_dim, const void* q_obs, const void* K);
ebd_status launch_score_mma(int units, int head_dim, int n_ctx, int n_obs, const void* q_obs,
                            const void* K, float* scores, float* lse, int32_t* dev_status,
                            cudaStream_t s);

}  // namespace ebd
