/*
 * ebd.h -- C ABI of the eviction-by-design (EBD) hot path on GB300 (sm_103a).
 *
 * Method: "Error Certificates for KV-Cache Eviction via Randomized Design"
 * (arXiv 2607.21475).  Per (batch row, KV head) unit the eviction step keeps
 * a certainty set A (attention sinks, a recency window, the score top slice),
 * draws a Poisson tail T = C \ A at known inclusion probabilities pi_i
 * (Section 3.3, Eq. 2) and compacts the survivors with one scalar
 * log(1/pi_i) each.  The certified decode step is Hajek-corrected attention
 * over the compact cache (Eq. 3) plus the design-based variance estimate
 * V_hat (Theorem 2) and the empirical-Bernstein radius r_t (Section 3.4,
 * Eq. 4), all from one pass over the compact cache.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Every pointer argument named as "device" is a CUDA device pointer into
 *   memory the caller owns (allocated by the caller, freed by the caller).
 *   The library never allocates, never frees, and keeps no pointer after the
 *   call returns.  `workspace` is caller-owned scratch of the size reported
 *   by the matching *_workspace_bytes query.
 * - `stream` is a cudaStream_t passed as void* (NULL = the legacy default
 *   stream).  Every call only enqueues work on it and returns: results are
 *   valid once the stream has been synchronised.  The tensor-core kernels of
 *   the certified decode (and its merge) are launched as programmatic
 *   dependents of whatever precedes them on the stream, and ebd_append lets
 *   what follows it launch early: a decode may start while its predecessor
 *   runs, but reads and writes memory only after that has completed, except
 *   for L2 prefetch hints (of its compact-cache rows and queries), which
 *   never change what a load returns.
 * - Tensors are dense, row-major, with the last dimension contiguous.
 *   B = batch, Hkv = KV heads, G = query heads per KV head (Hq = Hkv * G),
 *   d = head_dim, N = context length, cap = compact-cache capacity per unit.
 * - Argument errors are detected on the host and returned synchronously;
 *   nothing is enqueued in that case.  Data-dependent conditions found on
 *   the device are OR-ed into the caller's `dev_status` word (device int32,
 *   which the caller zeroes) as EBD_DEV_* bits; the call never traps,
 *   asserts or spins without a bound.
 * - dtype EBD_F32 or EBD_BF16 applies to K, V, Q, q_obs and the compact
 *   K_c, V_c; scores, pi, logw and every decode output are float32.
 */
#ifndef EBD_H_
#define EBD_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  EBD_OK = 0,
  EBD_ERR_INVALID = 1,     /* null pointer, non-positive or inconsistent size     */
  EBD_ERR_CAPACITY = 2,    /* capacity or workspace smaller than the call needs  */
  EBD_ERR_NONFINITE = 3,   /* reserved: non-finite scores are reported on device */
  EBD_ERR_UNSUPPORTED = 4, /* valid request outside what this build implements   */
  EBD_ERR_CUDA = 5         /* a CUDA runtime call or kernel launch failed        */
} ebd_status;

typedef enum { EBD_F32 = 0, EBD_BF16 = 1 } ebd_dtype;

/* Range term b_t of Eq. (4).  BOUND (default) is the one-pass triangle
 * inequality bound about a reference row c, the unit's middle retained row
 * V_c[(n - 1) / 2]:
 *   (max sqrt(1-pi) w ||v - c|| + ||y_hat - c|| max sqrt(1-pi) w) / N_hat,
 * never below the definition and, like it, unchanged when every value moves
 * by the same vector.  EXACT evaluates the definition
 * max_{S cap T} sqrt(1-pi_i) w_i ||v_i - y_hat|| / N_hat with a second pass over
 * the compact cache once y_hat is known. */
typedef enum { EBD_RANGE_BOUND = 0, EBD_RANGE_EXACT = 1 } ebd_range_mode;

/* Bits OR-ed into *dev_status by device code. */
#define EBD_DEV_CAPACITY 0x1  /* a unit kept more than `capacity` tokens; rows past
                                 capacity were dropped, n_kept holds the true count */
#define EBD_DEV_NONFINITE 0x2 /* a score was NaN or +-inf; that unit's output is
                                 unspecified (but every write stays in bounds)       */
#define EBD_DEV_TIMEOUT 0x4   /* an in-kernel pipeline wait hit its bound and the
                                 kernel returned early; outputs are unspecified      */

/* Tail design.  POISSON: independent Bernoulli(pi_i) draws (Section 3.3).
 * SYSTEMATIC: fixed-size systematic sampling at the same pi_i (Hajek 1964;
 * the exact-budget variant of Section 5): the tail in token order, cumulative
 * sums C_i of pi in units of 2^-32 (each pi_i rounded to the nearest unit),
 * one uniform u = (x >> 8) 2^-24 per unit with x = word 0 of Philox4x32-10 at
 * counter (2^32 - 1, kvh, layer, b); token i is kept when an integer lies in
 * (C_{i-1} - u, C_i - u].  Its inclusion probability is pi_i and the tail
 * sample has floor or ceil of sum pi tokens; joint inclusion probabilities do
 * not factor, so the certificate's variance form is then an approximation.
 * Supported at every context length (1 <= N <= 2^20). */
typedef enum { EBD_SAMPLING_POISSON = 0, EBD_SAMPLING_SYSTEMATIC = 1 } ebd_sampling;

/* Design of one layer's eviction (Section 3.3 and Appendix B of the paper). */
typedef struct {
  int32_t batch;         /* B                                                    */
  int32_t n_kv_heads;    /* Hkv                                                  */
  int32_t group;         /* G, query heads per KV head (used by scoring only)    */
  int32_t head_dim;      /* d                                                    */
  int32_t n_ctx;         /* N, cached tokens per unit, 1 <= N <= 2^20            */
  int32_t layer;         /* layer index: Philox counter word 2                   */
  uint64_t seed;         /* Philox key = (seed & 0xffffffff, seed >> 32)         */
  int32_t n_sink;        /* protected leading positions (attention sinks), 4     */
  int32_t n_recent;      /* protected trailing positions (recency window), 32    */
  int32_t k_head;        /* size of the score top slice (ties to lower index)    */
  int32_t budget_tokens; /* B_t: expected retained tokens per unit (A + tail)    */
  int32_t bisect_iters;  /* bisection steps for the scale c of Eq. (2), 1..200   */
  float eps;             /* probability floor, 1e-6 in the paper                 */
  int32_t sampling;      /* ebd_sampling of the tail (POISSON = 0)               */
} ebd_design;

/* Human-readable name of a status code (static string, never NULL). */
const char* ebd_status_string(ebd_status status);

/* ABI version of this library (increments on any signature change). */
int32_t ebd_abi_version(void);

/*
 * Failure-path check (no counterpart in the paper, which specifies no
 * runtime).  Launches one warp that waits, with the same bounded wait the
 * tensor-core pipelines use, on an mbarrier phase that nothing completes: the
 * wait gives up after ~2 s, the kernel raises EBD_DEV_TIMEOUT in *dev_status
 * (device int32, required; bits are OR-ed in) and returns, and the CUDA
 * context stays usable.  Lets a caller confirm that a stalled pipeline
 * reports a status instead of hanging the GPU.  Asynchronous on `stream`;
 * EBD_ERR_INVALID for a null dev_status.
 */
ebd_status ebd_check_stalled_wait(int32_t* dev_status, void* stream);

/*
 * Philox4x32-10 words used by the Poisson draw (Section 3.3: independent
 * Bernoulli(pi_i) retention on the tail).  For every unit (b, kvh) and token
 * i < N writes x0[b,kvh,i] (device uint32 [B,Hkv,N]) = output word i % 4 of
 * Philox4x32-10 (Salmon et al., SC'11) with key (seed_lo, seed_hi) and
 * counter (i / 4, kvh, layer, b): one generator call serves four consecutive
 * tokens.  The uniform the draw compares with pi_i is (x0 >> 8) * 2^-24.
 * Exposed so that the draws can be checked bit for bit.
 */
ebd_status ebd_philox_uniforms(uint64_t seed, int32_t layer, int32_t batch, int32_t n_kv_heads,
                               int32_t n_ctx, uint32_t* x0, void* stream);

/*
 * Accumulated-attention importance scores (Appendix B, harness: H2O-style
 * accumulated attention from observation queries).
 *   q_obs  device [B,Hkv,R,d] (dtype): the R = n_obs observation query rows
 *          of every query head of the KV head's group
 *   K      device [B,Hkv,N,d] (dtype)
 *   scores device [B,Hkv,N] float32 out: s_j = sum_r softmax_j(q_r . K^T / sqrt(d))
 * Needs workspace of ebd_score_workspace_bytes(B, Hkv, R) bytes.
 * Supports d in {64, 128}, 1 <= R <= 4096.
 */
size_t ebd_score_workspace_bytes(int32_t batch, int32_t n_kv_heads, int32_t n_obs);
ebd_status ebd_score(ebd_dtype dtype, int32_t batch, int32_t n_kv_heads, int32_t head_dim,
                     int32_t n_ctx, int32_t n_obs, const void* q_obs, const void* K,
                     float* scores, void* workspace, size_t ws_bytes, void* stream);

/*
 * Certainty set and inclusion probabilities (Section 3.3, Eq. 2).
 *   scores       device [B,Hkv,N] float32 importance scores
 *   pi           device [B,Hkv,N] float32 out: 1 on A; clip(c * s_i, eps, 1) on T
 *                with c such that sum_T pi_i = m = clamp(B_t - |A|, 0, |T|)
 *                (clip-saturated tokens join A; scores <= 0 sit at eps)
 *   certain_mask device [B,Hkv,N] uint8 out, nullable: 1 iff token in A
 *   dev_status   device int32, nullable: EBD_DEV_NONFINITE
 */
ebd_status ebd_compute_pi(const ebd_design* design, const float* scores, float* pi,
                          uint8_t* certain_mask, int32_t* dev_status, void* stream);

/*
 * Full eviction step of one layer (Section 3.3, Appendix B): certainty set,
 * Eq. (2) probabilities, Poisson draw, stable compaction.
 *   K, V      device [B,Hkv,N,d] (dtype)
 *   scores    device [B,Hkv,N] float32; or NULL together with q_obs
 *             (device [B,Hkv,n_obs,d]), in which case the scores are computed
 *             as by ebd_score
 *   K_c, V_c  device [B,Hkv,cap,d] (dtype) out: kept rows in increasing token order
 *   logw_c    device [B,Hkv,cap] float32 out: log(1/pi_i) of each kept row (0 on A)
 *   idx_c     device [B,Hkv,cap] int32 out: token index of each kept row
 *   n_kept    device [B,Hkv] int32 out: number of kept tokens (may exceed cap, in
 *             which case EBD_DEV_CAPACITY is raised and rows >= cap are dropped)
 *   dev_status device int32, required
 * Rows [n_kept, cap) of the outputs are left untouched.  Needs workspace of
 * ebd_evict_workspace_bytes(...) bytes (0 when scores are given).
 * Host-resident cache: with the scores given, K, V and the scores may be
 * page-locked host memory (cudaHostAlloc / cudaHostRegister, addressable by
 * the device): the select then reads every score and the gather only the kept
 * rows over the host link, instead of the whole cache being copied first.
 * Scoring (scores NULL) needs K and q_obs in device memory
 * (EBD_ERR_UNSUPPORTED otherwise).  Pageable host memory: EBD_ERR_INVALID.
 * Stream order: all work is ordered after earlier work on `stream` and
 * before later work on it.  With more units (B * Hkv) than SMs the call cuts
 * the units into chunks of one SM count and runs each chunk's select and
 * gather on its own stream (side streams of the library, one set per host
 * thread and device, created on the first such call made outside stream
 * capture), forked from and joined back into `stream` with events; this works
 * under stream capture and gives the same outputs as the single-stream order.
 */
size_t ebd_evict_workspace_bytes(const ebd_design* design, int32_t n_obs);
ebd_status ebd_evict(const ebd_design* design, ebd_dtype dtype, const void* K, const void* V,
                     const float* scores, const void* q_obs, int32_t n_obs, void* K_c, void* V_c,
                     float* logw_c, int32_t* idx_c, int32_t* n_kept, int32_t capacity,
                     int32_t* dev_status, void* workspace, size_t ws_bytes, void* stream);

/*
 * The two halves of ebd_evict, for callers that keep their own cache layout
 * (and for per-kernel timing).  ebd_evict(scores given) gives the outputs
 * of ebd_select then ebd_gather on the same stream.
 *
 * ebd_select: certainty set, Eq. (2) probabilities, Poisson draw and the
 * stable compaction of indices (Section 3.3, Appendix B) -- everything but
 * the row copy.
 *   scores  device [B,Hkv,N] float32
 *   idx_c   device [B,Hkv,cap] int32 out: kept token indices, increasing
 *   logw_c  device [B,Hkv,cap] float32 out: log(1/pi) of each kept token
 *   n_kept  device [B,Hkv] int32 out (may exceed cap: EBD_DEV_CAPACITY)
 *   dev_status device int32, required
 *
 * ebd_gather: copies rows K[idx_c[p]], V[idx_c[p]] to K_c[p], V_c[p] for
 * p < min(n_kept, cap) of every unit (16-byte loads; d * elem must be a
 * multiple of 16 bytes and the four tensors 16-byte aligned).  A row whose
 * index lies outside [0, n_ctx) is skipped (its K_c/V_c row is left as it
 * was), so a corrupt index list cannot make the copy read out of bounds.
 * The scores of ebd_select and K, V of ebd_gather may be page-locked host
 * memory, as for ebd_evict.
 */
ebd_status ebd_select(const ebd_design* design, const float* scores, int32_t* idx_c,
                      float* logw_c, int32_t* n_kept, int32_t capacity, int32_t* dev_status,
                      void* stream);
ebd_status ebd_gather(const ebd_design* design, ebd_dtype dtype, const void* K, const void* V,
                      const int32_t* idx_c, const int32_t* n_kept, int32_t capacity, void* K_c,
                      void* V_c, void* stream);

/*
 * One workspace size for a whole layer (the boundary of Section 3.1's problem
 * statement: the design fixed per layer, the retained set of `capacity` rows
 * per unit): the largest of ebd_evict_workspace_bytes(design, 0) (scores
 * given), ebd_evict_workspace_bytes(design, 64 * group) (accumulated-attention
 * scoring from 64 observation positions per query head, the window of
 * Appendix B) and ebd_decode_workspace_bytes(dtype, B, Hkv, G, d, capacity)
 * for either dtype.  A buffer of this size serves every call of the layer;
 * the per-call queries give exact, smaller sizes.  0 for a NULL design or
 * capacity < 1.  ebd_compute_pi, ebd_select and ebd_gather need none.
 */
size_t ebd_workspace_bytes(const ebd_design* design, int32_t capacity);

/*
 * Certified decode step (Eq. 3, Theorem 2, Eq. 4) for every query head.
 *   Q        device [B,Hkv*G,d] (dtype): query heads kvh*G .. kvh*G+G-1 read the
 *            compact cache of KV head kvh
 *   K_c,V_c  device [B,Hkv,cap,d] (dtype); logw_c device [B,Hkv,cap] float32
 *   n_kept   device [B,Hkv] int32 (values above cap are read as cap)
 *   delta    confidence parameter (0.1 in the paper); eps0 normaliser (1e-9)
 *   y        device [B,Hkv*G,d] float32 out: y_hat of Eq. (3)
 *   lse      device [B,Hkv*G] float32 out: log N_hat (-inf for an empty unit)
 *   var_hat  device [B,Hkv*G] float32 out: V_hat of Theorem 2
 *   b_t      device [B,Hkv*G] float32 out: range term (see ebd_range_mode)
 *   radius   device [B,Hkv*G] float32 out: r_t of Eq. (4)
 *   dev_status device int32, nullable
 * An empty unit (n_kept = 0) gives y = 0, lse = -inf and a zero certificate.
 * Needs workspace of ebd_decode_workspace_bytes(...) bytes for the split-K
 * partial records.  Supports d in {64, 128} and 1 <= G <= 16; a group of
 * more than 8 query heads is decoded in two slices of at most 8 heads, one
 * pass over the compact cache each (EBD_ERR_UNSUPPORTED beyond 16).
 * Results are reproducible bit for bit: a request always takes the same
 * kernels and the same summation order on a given GPU (the choice depends on
 * the request's shape and the GPU's SM count, so GPUs with another SM count
 * may differ in the last bits).
 */
size_t ebd_decode_workspace_bytes(ebd_dtype dtype, int32_t batch, int32_t n_kv_heads,
                                  int32_t group, int32_t head_dim, int32_t capacity);
ebd_status ebd_certified_decode(ebd_dtype dtype, int32_t batch, int32_t n_kv_heads, int32_t group,
                                int32_t head_dim, const void* Q, const void* K_c, const void* V_c,
                                const float* logw_c, const int32_t* n_kept, int32_t capacity,
                                float delta, float eps0, ebd_range_mode range_mode, float* y,
                                float* lse, float* var_hat, float* b_t, float* radius,
                                int32_t* dev_status, void* workspace, size_t ws_bytes,
                                void* stream);

/*
 * Certified decode that allocates nothing.  The paper has no counterpart: this
 * is a deployment variant of ebd_certified_decode for callers that cannot
 * allocate device memory -- serving stacks that lay out all device memory at
 * start-up and forbid cudaMalloc afterwards (an allocation can synchronise the
 * device and break a planned pool), and plugin hosts that give an operator its
 * inputs and outputs but no allocator.  Arguments, outputs and results are
 * those of ebd_certified_decode, without the workspace.
 *
 * The split-K scratch is a 16 MiB array inside the library (a static
 * __device__ variable, held by every GPU that loads the library until the
 * process exits).  The call allocates nothing and calls no allocating routine.
 * - Returns EBD_ERR_CAPACITY, before enqueueing anything, when the request
 *   needs more scratch than that (ebd_decode_workspace_bytes(...) > 16 MiB).
 * - The first call on each device looks up the array's device address with
 *   that device current (cudaGetSymbolAddress) and caches it; make that first
 *   call before any stream capture.
 * - Every call on a device shares the one array, which keeps the previous
 *   call's contents (nothing in it needs to start at zero).  Calls whose work
 *   overlaps on the GPU -- unordered streams, or several host threads -- race
 *   on it; the caller must order them.
 */
ebd_status ebd_certified_decode_static(ebd_dtype dtype, int32_t batch, int32_t n_kv_heads,
                                       int32_t group, int32_t head_dim, const void* Q,
                                       const void* K_c, const void* V_c, const float* logw_c,
                                       const int32_t* n_kept, int32_t capacity, float delta,
                                       float eps0, ebd_range_mode range_mode, float* y,
                                       float* lse, float* var_hat, float* b_t, float* radius,
                                       int32_t* dev_status, void* stream);

/*
 * Decode-time growth of a compact cache: one new token per unit joins the
 * cache with pi = 1 (log(1/pi) = 0), as every token generated after an
 * eviction is kept until the next one.  For each unit with n_kept < capacity,
 * row n_kept of K_c/V_c receives k_new/v_new, logw_c gets 0 and idx_c the
 * token position; n_kept grows by one.  A full unit keeps its rows, counts the
 * token in n_kept anyway and raises EBD_DEV_CAPACITY (as eviction overflow).
 *   k_new, v_new  device [B,Hkv,d] (dtype), 16-byte aligned
 *   positions     device [B] int32: position of the new token of each row
 *   K_c, V_c, logw_c, idx_c, n_kept, capacity: the compact cache (updated)
 *   dev_status    device int32, required
 */
ebd_status ebd_append(ebd_dtype dtype, int32_t batch, int32_t n_kv_heads, int32_t head_dim,
                      const void* k_new, const void* v_new, const int32_t* positions, void* K_c,
                      void* V_c, float* logw_c, int32_t* idx_c, int32_t* n_kept,
                      int32_t capacity, int32_t* dev_status, void* stream);

/*
 * Re-eviction of a resident compact cache: the tail draws redrawn every T_r
 * decode steps (the block schedule of the anytime argument, Section 4 and its
 * appendix).  Each unit's resident rows (the first min(n_kept_in, cap_in)
 * rows, in cache order) are the context of a new eviction with `design`:
 * certainty set (the first n_sink and last n_recent resident rows, the
 * k_head highest scores), Eq. (2) probabilities on the tail, Poisson draws
 * keyed by (design->seed; resident position / 4, kvh, design->layer, b) -- pass
 * a fresh seed per round -- and compaction.  A token kept by both rounds has
 * inclusion probability pi_1 pi_2 (the two Poisson designs compose), so the
 * output log(1/pi) is logw_in + log(1/pi_2), and idx_out holds the original
 * token positions (idx_in of the kept rows).
 *   design->n_ctx must equal cap_in (the row stride of scores and the inputs)
 *   scores        device [B,Hkv,cap_in] float32: importance of the resident rows
 *   K_in, V_in, logw_in, idx_in, n_kept_in, cap_in: the resident cache (read)
 *   K_out, V_out, logw_out, idx_out, n_kept_out, cap_out: the new cache;
 *                 distinct from the inputs (EBD_ERR_INVALID otherwise)
 *   dev_status    device int32, required (EBD_DEV_CAPACITY, EBD_DEV_NONFINITE)
 */
ebd_status ebd_reevict(const ebd_design* design, ebd_dtype dtype, const float* scores,
                       const void* K_in, const void* V_in, const float* logw_in,
                       const int32_t* idx_in, const int32_t* n_kept_in, int32_t cap_in,
                       void* K_out, void* V_out, float* logw_out, int32_t* idx_out,
                       int32_t* n_kept_out, int32_t cap_out, int32_t* dev_status, void* stream);

/*
 * Observation queries for E0 (Appendix, experimental details: accumulated
 * attention from strided prefill queries, a SnapKV-style window of the last 64
 * prefill positions, or question-position queries).  Copies the prefill query
 * rows at `positions` into the observation layout ebd_score reads:
 *   q_obs[b, kvh, g * P + p, :] = Q[b, kvh * G + g, positions[p], :]
 *   Q         device [B, Hkv*G, n_rows_q, d] (dtype), 16-byte aligned
 *   positions device [P] int32, each in [0, n_rows_q) (not checked on device)
 *   q_obs     device [B, Hkv, G*P, d] (dtype) out
 */
ebd_status ebd_gather_queries(ebd_dtype dtype, int32_t batch, int32_t n_kv_heads, int32_t group,
                              int32_t head_dim, int32_t n_rows_q, const void* Q,
                              const int32_t* positions, int32_t n_pos, void* q_obs,
                              void* stream);

/*
 * Per-token variance contributions: the terms of Theorem 2's estimator,
 *   contrib[b, h, i] = (1 - pi_i) p_i^2 ||v_i - y_hat_h||^2,  p_i = w_i / N_hat,
 * so that sum_i contrib[b, h, i] = V_hat of head h.  Certain rows (pi = 1) and
 * rows at or past min(n_kept, cap) get 0.  A second pass over the compact
 * cache after ebd_certified_decode, whose y and lse it reads (Section 5's
 * fine-grained probe records these per retained token).
 *   Q, K_c, V_c, logw_c, n_kept, capacity: as for ebd_certified_decode
 *   y, lse     device [B, Hkv*G, d] / [B, Hkv*G] float32 from the decode
 *   contrib    device [B, Hkv*G, capacity] float32 out
 * Supports d in {64, 128} and G <= 8.
 */
ebd_status ebd_variance_contributions(ebd_dtype dtype, int32_t batch, int32_t n_kv_heads,
                                      int32_t group, int32_t head_dim, const void* Q,
                                      const void* K_c, const void* V_c, const float* logw_c,
                                      const int32_t* n_kept, int32_t capacity, const float* y,
                                      const float* lse, float* contrib, void* stream);

/*
 * Block scores for contribution-guided retrieval (Section 5, finer grains):
 * for every block k of `block` original positions, the sum over the unit's G
 * query heads of the contributions of its retained rows with idx_c in
 * [k * block, (k + 1) * block) -- the blocks whose evicted tokens sit among
 * high-contribution retained neighbours rank first.  Deterministic order.
 *   contrib  device [B, Hkv*G, capacity] from ebd_variance_contributions
 *   idx_c, n_kept, capacity: the compact cache (idx_c increasing per unit)
 *   out      device [B, Hkv, n_blocks] float32
 */
ebd_status ebd_block_scores(int32_t batch, int32_t n_kv_heads, int32_t group,
                            const float* contrib, const int32_t* idx_c, const int32_t* n_kept,
                            int32_t capacity, int32_t block, int32_t n_blocks, float* out,
                            void* stream);

/*
 * Deployed certificate and red-flag rule (the experimental setup of Section 5
 * and its appendix; the rule cert >= tau = 1 of Section 5).  At each of the
 * first six decode steps the radii r_t of Eq. (4) (delta = 0.1) of every
 * `head_stride`-th query head (4 in the paper) of every layer are averaged per
 * sequence; the certificate is the maximum of those step averages.  Call once
 * per probed step, after that step's certified decodes of all layers.
 *   radius      device [L, B, Hq] float32: the step's r_t, layer-major (pass
 *               radius + l * B * Hq as the radius output of layer l's decode)
 *   head_stride query heads h with h % head_stride == 0 enter the average
 *   tau         red-flag threshold (1 in the paper)
 *   first_step  nonzero: cert = this step's average (no earlier value is read)
 *   step_mean   device [B] float32 out, nullable: this step's average
 *   cert        device [B] float32 in/out: maximum over the probed steps so far
 *   red_flag    device [B] int32 out, nullable: 1 when cert >= tau
 * The average of each row is summed in a fixed order (deterministic).
 */
ebd_status ebd_certificate_update(const float* radius, int32_t n_layers, int32_t batch,
                                  int32_t n_q_heads, int32_t head_stride, float tau,
                                  int32_t first_step, float* step_mean, float* cert,
                                  int32_t* red_flag, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* EBD_H_ */
