/*
 * gmc.h -- C ABI of the GB300 library for one Global Momentum Compression
 * (GMC / GMC+) step, with K data-parallel workers simulated on one GPU.
 *
 * Method: Shi et al., "Global Momentum Compression for Sparse Communication in
 * Distributed Learning", arXiv 1905.12948.
 *   Algorithm 1 (GMC, Sec. 3.1), for every worker k and step t:
 *     e_{t+1/2,k} = e_{t,k} + g_{t,k} - (beta/eta) (w_t - w_{t-1})
 *     send C(e_{t+1/2,k});  e_{t+1,k} = e_{t+1/2,k} - C(e_{t+1/2,k})
 *     w_{t+1} = w_t - (eta/K) sum_k C(e_{t+1/2,k})
 *   with w_{-1} = w_0 and e_{0,k} = 0.
 *   Algorithm 2 (GMC+, Sec. 4) adds the detached point
 *     w_{t+1,k} = w_{t+1} - lambda*eta*e_{t+1,k}.
 *   Compressors (Sec. 4, Sec. 5.1, Sec. 5.2): exact top-s ("top-k"), the
 *   approximate top-s of Sec. 5.1 (a threshold taken from a random sample),
 *   and RBGS (random blocks chosen with one seed shared by all workers).
 *
 * Arithmetic: fp32, one IEEE round-to-nearest-even rounding per operation in
 * the order written above: v = (e + g) - (c * (w_t - w_{t-1})), c = fl(beta/eta);
 * the aggregate adds the workers' values in ascending worker order starting
 * from +0; w_{t+1} = w_t - (a * sum), a = fl(eta/K); detach w - (b * e),
 * b = fl(lambda*eta). Top-k ranks |v| through the fp32 bit pattern with the
 * sign cleared; ties go to the lower index. k = max(1, floor(ratio*d)).
 *
 * Conventions (all calls):
 *   - Every pointer argument named *_dev is device memory on the GPU that was
 *     current when the handle was created; *_host arguments are host memory.
 *   - The library owns its state (w, w_{t-1} - w_t, residuals, workspace),
 *     allocated once in gmc_create and freed in gmc_destroy. Caller buffers
 *     are borrowed: they must stay valid until the stream has passed the call.
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream). Calls are
 *     stream-ordered and asynchronous unless marked "synchronising".
 *   - Argument errors return at once and enqueue nothing. Data-dependent
 *     errors (a non-finite accumulator value, an internal consistency check)
 *     are recorded in a device status word read by gmc_check.
 *   - A handle is not thread-safe; distinct handles are independent.
 *   - No C++ exception crosses this boundary.
 */
#ifndef GMC_H
#define GMC_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct gmc_ctx* gmc_t;

/* Status codes. */
#define GMC_OK          0  /* success */
#define GMC_EINVAL      1  /* invalid argument or handle */
#define GMC_ENOMEM      2  /* device or host allocation failed */
#define GMC_ECUDA       3  /* a CUDA call or kernel launch failed */
#define GMC_ENONFINITE  4  /* a step met a NaN or Inf accumulator value */
#define GMC_ESTATE      5  /* call out of order (e.g. gmc_step before gmc_set_params) */
#define GMC_EINTERNAL   6  /* an internal consistency check failed on the device */
#define GMC_ETOOBIG     7  /* size above the fixed scratch of gmc_topk_noalloc */
#define GMC_ETIMEOUT    8  /* a bounded wait in a step's kernel gave up: work was skipped */

/* Compressors C(.). */
#define GMC_TOPK 0 /* exact top-k by magnitude, ties to the lower index (Sec. 4 top-s) */
#define GMC_RBGS 1 /* random aligned blocks of `block` components (Sec. 4, Sec. 5.2) */
#define GMC_TOPK_APPROX 2 /* approximate top-s (Sec. 5.1): a sample S of about d/100
                             components -- n = max(1, floor(d/800)) runs of 8
                             consecutive ones, one per stratum [floor(i d/n),
                             floor((i+1) d/n)) starting on a multiple of 8 picked by
                             the SplitMix64 stream of (seed, t), drawn afresh each
                             step and shared by all workers (d < 8: all of [0, d)) --
                             gives theta, the r-th largest sampled |v| with
                             r = max(1, floor(ratio*|S|)); every component with
                             |v| >= theta is sent (the count varies), unless more
                             than min(d, 4 s + 4096) do (s = max(1, floor(ratio*d))):
                             then the exact top of that many */

/* Variants of the step (gmc_set_variant): the method, and the appendix's other
 * ways to combine momentum with error feedback, for comparison. */
#define GMC_VARIANT_GMC              0 /* Alg. 1 (default) */
#define GMC_VARIANT_SERVER_MOMENTUM  1 /* Alg. 3: e_{t+1/2,k} = e_{t,k} + g_{t,k};
                                          w_{t+1} = (w_t - (eta/K) sum_k C_k)
                                                    + beta (w_t - w_{t-1}), a dense update */
#define GMC_VARIANT_LR_IN_RESIDUAL   2 /* Alg. 4: e_{t+1/2,k} = (e_{t,k} + eta g_{t,k})
                                                             - beta (w_t - w_{t-1});
                                          w_{t+1} = w_t - fl(1/K) sum_k C_k */
/* The local-momentum baseline the paper compares against (Sec. 2.3 eq. (3) with
 * error feedback; DGC without / with momentum factor masking, Sec. 3.1):
 *   m_{t+1,k} = beta m_{t,k} + eta g_{t,k} (m_{0,k} = 0), e_{t+1/2,k} = e_{t,k} + m_{t+1,k},
 *   w_{t+1} = w_t - fl(1/K) sum_k C_k; with masking, m_{t+1,k} = 0 where worker k sent.
 *   Its detached point (DEF-A-like, lambda > 0) is w_{t,k} = w_t - lambda e_{t,k}. */
#define GMC_VARIANT_LOCAL_MOMENTUM      3
#define GMC_VARIANT_LOCAL_MOMENTUM_MFM  4

/* Top-k selection engines; both give identical results. */
#define GMC_SELECT_SAMPLED 0 /* default: a sampled threshold filters candidates in the one
                                dense pass; exact radix select among them; falls back to
                                GMC_SELECT_DENSE for a worker whose filter missed */
#define GMC_SELECT_DENSE   1 /* exact multi-pass radix select over the dense accumulator */

/* Slots of the counters returned by gmc_get_stats and gmc_step_host. */
#define GMC_STAT_STEPS      0 /* steps taken (cumulative counters only) */
#define GMC_STAT_PAIRS      1 /* sum_k |supp C_k|: components sent by the workers */
#define GMC_STAT_NNZ        2 /* sum_k ||C_k||_0: sent components that are non-zero */
#define GMC_STAT_UNION      3 /* |U_t|: coordinates sent by at least one worker */
#define GMC_STAT_CHANGED    4 /* ||w_{t+1} - w_t||_0 */
#define GMC_STAT_FALLBACKS  5 /* workers whose sampled filter fell back to the dense select */
#define GMC_STAT_NONFINITE  6 /* accumulator values that were NaN or Inf */
#define GMC_STAT_COUNT      8 /* array length to pass */

/* Kernel ids for gmc_profile_read. */
#define GMC_KERNEL_ACCUMULATE  0 /* fused accumulator + candidate filter (top-k), one dense pass */
#define GMC_KERNEL_RBGS_STEP   1 /* fused accumulator + RBGS compress + aggregate + update */
#define GMC_KERNEL_SAMPLE      2 /* sampled threshold per worker */
#define GMC_KERNEL_SELECT      3 /* exact select among candidates (2 launches per step) */
#define GMC_KERNEL_DENSE       4 /* exact dense select for workers that fell back */
#define GMC_KERNEL_COMPACT     5 /* reserved: no launch (the dense pass writes C(v) as
                                    index-ordered sub-chunks) */
#define GMC_KERNEL_AGGREGATE   6 /* marks the sent pairs; when the aggregation is not
                                    deferred also the worker-ordered aggregate + update */
#define GMC_KERNEL_RBGS_PICK   7 /* RBGS block choice (Floyd sampling) */
#define GMC_KERNEL_DETACH      8 /* GMC+ detached points */
#define GMC_KERNEL_OTHER       9 /* counters and small bookkeeping */
#define GMC_KERNEL_COUNT      10

/*
 * gmc_create -- allocate a handle and its device state on the current device.
 * Inputs of Algorithm 1 (Sec. 3.1): d parameters, K workers, momentum beta in
 * [0,1), learning rate eta > 0, compressor C; ratio in (0,1] is the kept share
 * (top-k: k = max(1, floor(ratio*d)); RBGS: m = max(1, floor(ratio*nb)) of the
 * nb = ceil(d/block) blocks; approximate top-s: ratio*|S| sampled components
 * reach theta); block >= 1 is the RBGS block size (ignored otherwise).
 * Requires 1 <= d < 2^31 - 2^16 and 1 <= K <= 32.
 * GMC+'s lambda defaults to 0 (plain GMC) for top-k and 0.5 for RBGS (Sec. 5.2
 * uses 0.5 for GMC+). Returns GMC_EINVAL, GMC_ENOMEM or GMC_ECUDA on failure,
 * with *out set to NULL. The state must be initialised with gmc_set_params.
 */
int gmc_create(gmc_t* out, int64_t d, int32_t K, float beta, float eta,
               int32_t compressor, double ratio, int64_t block);

/* gmc_destroy -- synchronise the device and free everything the handle owns: the
 * state Alg. 1 (Sec. 3.1) carries between steps (w_t, w_t - w_{t-1}, the K
 * residuals e_{t,k}) and the workspace. NULL is ignored. Returns nothing; after
 * it, h must not be used. */
void gmc_destroy(gmc_t h);

/* gmc_set_lambda -- GMC+ detach coefficient lambda in [0,1] (Alg. 2); 0 is GMC.
 * GMC_EINVAL for lambda != 0 under Alg. 3 / Alg. 4 (GMC+ detaches Alg. 1); the
 * local-momentum baseline detaches as w_t - lambda e_{t,k}. */
int gmc_set_lambda(gmc_t h, float lambda);

/* gmc_set_rbgs_mode -- 0: one block choice per step shared by all workers, as in
 * Sec. 4 / Sec. 5.2 (default); 1: an independent choice per worker. */
int gmc_set_rbgs_mode(gmc_t h, int32_t per_worker);

/* gmc_set_seed -- seed of the RBGS block choice (SplitMix64 counter stream
 * keyed by (seed, t[, k]); Floyd's sampling) and of the approximate top-s
 * sample (the stream of (seed, t)). Default 0. */
int gmc_set_seed(gmc_t h, uint64_t seed);

/* gmc_set_eta -- change eta between steps (e.g. the cosine schedule of Sec. 5.1);
 * takes effect at the next gmc_step. */
int gmc_set_eta(gmc_t h, float eta);

/* gmc_set_variant -- the step's form (GMC_VARIANT_*; default Alg. 1). Only for the
 * top-k compressors (exact and approximate), with lambda = 0 for Alg. 3 / Alg. 4,
 * and only before the first step after gmc_create or gmc_set_params (GMC_ESTATE
 * otherwise), since the residuals mean another thing under each form.
 * GMC_VARIANT_SERVER_MOMENTUM allocates d floats of w_t - w_{t-1} and turns off
 * the deferred aggregation: every step ends with a dense pass over w. The
 * local-momentum variants allocate K x d floats of momentum (read and written
 * by every step's dense pass); masking turns off the deferred aggregation.
 * GMC_ENOMEM if an allocation fails; synchronising when it allocates.
 * Arithmetic: each operation rounded once, in the order written beside the
 * GMC_VARIANT_* constants. */
int gmc_set_variant(gmc_t h, int32_t variant);

/* gmc_set_select_mode -- GMC_SELECT_SAMPLED (default) or GMC_SELECT_DENSE (exact
 * top-k only: GMC_EINVAL for GMC_TOPK_APPROX, which its sample defines). */
int gmc_set_select_mode(gmc_t h, int32_t mode);

/* gmc_set_detach_output -- GMC+ (Alg. 2 detach): when out_dev is not NULL, every
 * following gmc_step also writes w_{t+1,k} = w_{t+1} - lambda*eta*e_{t+1,k} into
 * out_dev[k*ld + j] (K rows, row stride ld >= d floats, caller-owned and borrowed
 * until disabled with NULL). */
int gmc_set_detach_output(gmc_t h, float* out_dev, int64_t ld);

/* gmc_set_params -- w_0 := w0_dev[0..d) (device, fp32); also sets w_{-1} = w_0,
 * e_{0,k} = 0, t = 0 and clears the counters (Alg. 1 initialisation). */
int gmc_set_params(gmc_t h, const float* w0_dev, void* stream);

/* gmc_step -- one iteration t of Alg. 1 (Alg. 2 when lambda > 0 and a detach
 * output is set). grads_dev: K x d fp32, row-major (worker k's gradient
 * g_{t,k} at grads_dev[k*d .. k*d+d)), device memory, read-only, borrowed until
 * the stream has passed the step; any alignment. Enqueues kernels only; never
 * synchronises. Non-finite accumulator values still complete the step
 * deterministically and are reported by gmc_check as GMC_ENONFINITE.
 *
 * Deferred aggregation (top-k with d >= 4096 * 2 * SMs, about 1.25 M on GB300):
 * the step selects and records C(e_{t+1/2,k}) but leaves the last line of
 * Alg. 1 -- w_{t+1} = w_t - (eta/K) sum_k C_k and the zeroing of the sent
 * residuals -- to the next gmc_step, whose single pass over the tiles applies
 * it before forming its own accumulator. The results are the same, bit for
 * bit: every call that reads the state (gmc_get_params, gmc_get_residual,
 * gmc_get_worker_params, gmc_get_stats) first applies a pending aggregation,
 * on its own stream after the step. gmc_step_host and a set detach output
 * apply it within the step. Because a getter writes the state, a getter on
 * one stream and a later gmc_step on another are ordered by the library. */
int gmc_step(gmc_t h, const float* grads_dev, void* stream);

/* gmc_step_host -- gmc_step from host memory grads_host (K x d fp32,
 * row-major), borrowed until the stream has passed the call. Page-locked
 * (pinned) host memory is read in place by the step's kernels over the host
 * link; other host memory is first copied into a library staging buffer
 * (allocated on the first such call). The step's aggregation is applied
 * within the call, and its counters (GMC_STAT_COUNT uint64 slots,
 * GMC_STAT_STEPS slot = 1) are copied into step_stats_host, which must then be
 * pinned host memory valid until the stream has passed the call (or NULL to
 * skip the read-back). */
int gmc_step_host(gmc_t h, const float* grads_host, uint64_t* step_stats_host, void* stream);

/* gmc_step_bf16 / gmc_step_host_bf16 -- gmc_step / gmc_step_host with the
 * gradients in bfloat16: K x d row-major 16-bit values, each the upper half of
 * an fp32 bit pattern, widened exactly to fp32 as they are read (the step's
 * arithmetic is unchanged). Halves the gradient bytes the step reads (device)
 * or moves over the host link (host). The pointer must be 2-byte aligned
 * (GMC_EINVAL otherwise); ownership, ordering and errors as gmc_step /
 * gmc_step_host. */
int gmc_step_bf16(gmc_t h, const uint16_t* grads_bf16_dev, void* stream);
int gmc_step_host_bf16(gmc_t h, const uint16_t* grads_bf16_host, uint64_t* step_stats_host,
                       void* stream);

/* gmc_get_params -- copy the server's parameters w_t of Alg. 1 (Sec. 3.1; the
 * w_{t+1} = w_t - (eta/K) sum_k C_k line of the last step applied), d floats, into
 * w_dev_out (device, caller-owned, borrowed until the stream has passed the
 * call), applying a pending aggregation first (see gmc_step). GMC_EINVAL for a
 * NULL pointer, GMC_ESTATE before gmc_set_params. */
int gmc_get_params(gmc_t h, float* w_dev_out, void* stream);

/* gmc_get_residual -- copy worker k's residual e_{t,k} = e_{t-1/2,k} - C(e_{t-1/2,k})
 * of Alg. 1 (Sec. 3.1; +0 exactly where the worker sent), d floats, into
 * e_dev_out (device, caller-owned, borrowed until the stream has passed the
 * call), applying a pending aggregation first. GMC_EINVAL for k outside [0, K)
 * or a NULL pointer, GMC_ESTATE before gmc_set_params. */
int gmc_get_residual(gmc_t h, int32_t k, float* e_dev_out, void* stream);

/* gmc_get_selected -- synchronising. The last step's C(e_{t-1/2,k}) of worker k
 * as (index, value) pairs in ascending index order: *count_host pairs written to
 * idx_dev / val_dev (device, capacity entries each). Returns GMC_EINVAL if
 * capacity is too small (with *count_host set to the size needed), GMC_ESTATE
 * before the first step. */
int gmc_get_selected(gmc_t h, int32_t k, uint32_t* idx_dev, float* val_dev,
                     int64_t capacity, int64_t* count_host, void* stream);

/* gmc_selected_capacity -- the largest number of pairs one worker can send per
 * step (k for top-k, min(d, 4 s + 4096) for the approximate top-s, m*block for
 * RBGS), or -1 for an invalid handle. */
int64_t gmc_selected_capacity(gmc_t h);

/* gmc_get_worker_params -- GMC+ detached point of worker k at the current step,
 * w_{t,k} = w_t - lambda*eta*e_{t,k} (Alg. 2), written to out_dev (d floats). */
int gmc_get_worker_params(gmc_t h, int32_t k, float* out_dev, void* stream);

/* gmc_get_stats -- synchronising (applies a pending aggregation first, on a
 * library stream ordered after the last step). Cumulative counters since gmc_set_params
 * (n <= GMC_STAT_COUNT slots copied into counters_host) and the relative
 * communication cost of Sec. 5, RCC = (K*sum_t ||w_{t+1}-w_t||_0 +
 * sum_t sum_k ||C_k||_0) / (d K T), halved for RBGS (no indices, Sec. 5.2). */
int gmc_get_stats(gmc_t h, uint64_t* counters_host, int32_t n, double* rcc_host);

/* Checkpoint / resume. A saved state is the handle's state between steps as
 * Alg. 1 defines it (any pending aggregation applied first): w_t,
 * w_t - w_{t-1}, every residual e_{t,k}, Alg. 3's server momentum, the step t,
 * eta, seed, lambda, the RBGS mode, the selection engine and the cumulative
 * counters, behind a fixed header (magic "GMCSTATE", version 1) holding d, K,
 * the compressor, ratio, block and variant. Host memory, little-endian fp32.
 *
 * gmc_state_bytes -- bytes gmc_save_state writes for this handle (-1: invalid
 * handle). */
int64_t gmc_state_bytes(gmc_t h);

/* gmc_save_state -- synchronising. Writes gmc_state_bytes(h) bytes to host_out
 * (any host memory, capacity bytes). GMC_EINVAL if capacity is too small,
 * GMC_ESTATE before gmc_set_params. */
int gmc_save_state(gmc_t h, void* host_out, int64_t capacity);

/* gmc_load_state -- synchronising. Replaces the handle's state with a saved one
 * (bytes long). The handle must have been created with the same d, K,
 * compressor, ratio (and block for RBGS) and set to the same variant: else, or
 * for a malformed buffer, GMC_EINVAL and the state is left as it was. The next
 * gmc_step continues the saved trajectory exactly (it reads w_t - w_{t-1}
 * densely once, as no pair lists of the step before were saved);
 * gmc_get_selected returns GMC_ESTATE until that step. */
int gmc_load_state(gmc_t h, const void* host_in, int64_t bytes);

/* gmc_check -- synchronising. Reports what the device recorded since gmc_set_params
 * (or gmc_load_state), most severe first: GMC_ECUDA (a CUDA error, e.g. a failed
 * kernel), GMC_EINTERNAL (an internal consistency check failed), GMC_ETIMEOUT (a
 * bounded wait of a bulk pass gave up, about two seconds without progress, and the
 * pass skipped the rest of that CTA's tiles: w and the residuals are not Alg. 1's
 * and the handle must be reset with gmc_set_params or gmc_load_state), or
 * GMC_ENONFINITE (a NaN or Inf accumulator value, Sec. 3.1's step otherwise
 * completed). GMC_OK when none. The status is not cleared by reading it.
 * The recorded state is Alg. 1's (Sec. 3.1): the step runs to completion or
 * says which condition it met; the paper itself defines no error behaviour. */
int gmc_check(gmc_t h);

/* gmc_profile_enable -- when on, each kernel launch of gmc_step is bracketed by
 * CUDA events on the step's stream; gmc_profile_read reports the totals. */
int gmc_profile_enable(gmc_t h, int32_t on);

/* gmc_profile_kernels -- which launches gmc_profile_enable brackets: bit k of
 * kernel_mask selects kernel id k (GMC_KERNEL_*); default all. Each bracketed
 * launch costs two event records on the stream, so timing only the kernels of
 * interest keeps the step's own time undisturbed. */
int gmc_profile_kernels(gmc_t h, uint32_t kernel_mask);

/* gmc_profile_read -- synchronising. For kernel id `kernel` (GMC_KERNEL_*): the
 * summed device time in ms, the number of launches, and the algorithmic bytes
 * those launches had to move (the minimum traffic of the operation), since
 * profiling was enabled. Resets nothing. */
int gmc_profile_read(gmc_t h, int32_t kernel, double* total_ms, int64_t* launches,
                     double* algorithmic_bytes);

/* gmc_kernel_name -- a static name for a GMC_KERNEL_* id ("?" if unknown). */
const char* gmc_kernel_name(int32_t kernel);

/*
 * Failure injection for tests. The paper has no counterpart: these exist so
 * that the library's failure paths can be exercised without faulting a GPU.
 *
 * gmc_test_fail_alloc -- process-wide. With fail_at >= 0, the fail_at-th device
 * allocation the library makes from now on (0 = the next one, by any handle)
 * fails as cudaMalloc does when memory runs out, once; fail_at < 0 disarms it.
 * Returns the number of device allocations all handles hold at the call, so a
 * test can check that a failed gmc_create or gmc_set_variant leaks nothing.
 */
int64_t gmc_test_fail_alloc(int64_t fail_at);

/*
 * gmc_test_withhold_copy -- the next gmc_step of h (only that one) runs its bulk
 * pass with the copy of one item, worker k's slice of tile `tile` (4096
 * components from tile*4096), never issued, and with every wait of that pass
 * bounded by wait_limit_ns (1 .. 2e9) instead of about two seconds. The waits on
 * that item give up, the CTA skips its remaining tiles after the copies it did
 * issue have landed, and gmc_check then reports GMC_ETIMEOUT. GMC_EINVAL when
 * the handle's step has no bulk pass (exact or approximate top-k needs
 * d >= 4096 * 2 * SMs and K <= 16; RBGS d >= 4096 * SMs), or for a tile, worker or
 * limit out of range.
 */
int gmc_test_withhold_copy(gmc_t h, int64_t tile, int32_t k, uint64_t wait_limit_ns);

/*
 * gmc_topk_noalloc -- the top-k compressor of one vector without allocating.
 * The paper has no counterpart: this is a library convenience for callers
 * that cannot call cudaMalloc, e.g. code whose device memory is all owned by
 * another allocator (a framework's caching pool or a fixed serving budget),
 * so neither the library nor the caller may allocate scratch for it.
 * Writes the k pairs (index, value) of x_dev[0..n) that come first under
 * (|x| fp32 bit pattern descending, index ascending) -- the same selection as
 * GMC_TOPK -- to idx_dev / val_dev (device, k entries each) in ascending index
 * order. x_dev is device memory, fp32, read-only. Requires 1 <= k <= n
 * (else GMC_EINVAL) and n <= 2^26 (else GMC_ETOOBIG).
 * It allocates nothing: its scratch is one fixed array of about 270 KB in the
 * library's device memory, which every GPU that loads the library holds until
 * the process exits. All calls share that array, so calls that overlap on the
 * GPU (on different streams, or from different threads) race; serialise
 * them. The first call on each device (and the first after the device's
 * context was replaced, e.g. by cudaDeviceReset) looks up the array's device
 * address and the SM count; make that first call before any stream capture.
 * A NaN in x ranks above every finite value and Inf (its magnitude bit pattern
 * is larger) and is not reported as an error. Stream-ordered, asynchronous;
 * GMC_ECUDA if a launch fails (only that launch's error is reported).
 */
int gmc_topk_noalloc(const float* x_dev, int64_t n, int64_t k, uint32_t* idx_dev, float* val_dev,
                     void* stream);

/* gmc_strerror -- a static message for a status code. */
const char* gmc_strerror(int status);

#ifdef __cplusplus
}
#endif

#endif /* GMC_H */
