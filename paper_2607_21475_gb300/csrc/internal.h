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

// Design validation shared by the eviction entry points (evict.cu).
ebd_status check_design(const ebd_design* d);

// E1-E4a for every unit (evict.cu): certainty set, pi, draws, index
// compaction.  n_len (nullable, device [units]) gives each unit's context
// length when it is below the row stride d->n_ctx of `scores`.
ebd_status launch_select(const ebd_design* d, const float* scores, const int32_t* n_len,
                         float* pi, uint8_t* mask, int32_t* idx_c, float* logw_c, int32_t* n_kept,
                         int cap, int32_t* dev_status, cudaStream_t stream);

// E4b for every unit (evict.cu): rows K[idx_c[p]], V[idx_c[p]] (row stride
// d->n_ctx) to K_c[p], V_c[p] for p < min(n_kept, cap); rows whose index lies
// outside [0, n_ctx) are skipped.
ebd_status launch_gather(const ebd_design* d, ebd_dtype dtype, const void* K, const void* V,
                         const int32_t* idx_c, const int32_t* n_kept, int cap, void* K_c,
                         void* V_c, cudaStream_t s);

// The same for the units [unit0, unit0 + n_units) only.  `ctas_per_unit`:
// the cluster size of the shared-memory select (0: chosen for this launch's
// units; a caller that splits one request into several launches passes the
// size chosen for the whole request, so each unit is split the same way).
ebd_status launch_select_range(const ebd_design* d, const float* scores, const int32_t* n_len,
                               float* pi, uint8_t* mask, int32_t* idx_c, float* logw_c,
                               int32_t* n_kept, int cap, int32_t* dev_status, int unit0,
                               int n_units, cudaStream_t stream, int ctas_per_unit);

// CTAs per unit of the shared-memory select for `units` units of n_ctx
// tokens (0 when the context is too long for a cluster).
int select_cluster_size(int n_ctx, int units);
ebd_status launch_gather_range(const ebd_design* d, ebd_dtype dtype, const void* K,
                               const void* V, const int32_t* idx_c, const int32_t* n_kept,
                               int cap, void* K_c, void* V_c, int unit0, int n_units,
                               cudaStream_t s);

bool aligned16(const void* p);

// Address under which kernels read a caller's buffer: device or managed memory
// as is, page-locked host memory through its device mapping (read over the
// host link); nullptr for memory the device cannot address (evict.cu).
const void* device_address(const void* p);
bool is_device_memory(const void* p);

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
