/*
 * barycache.h -- C ABI of the GB300 (sm_103a) BaryCache skipped-step forecast library.
 *
 * BaryCache (Barycentric Extrapolator, Sec. 3.2-3.3) accelerates DiT sampling by running
 * the full model only on some diffusion steps ("full steps") and predicting the cached
 * features on the others ("skipped steps" / cache forward) as a fixed linear combination
 * of the H most recent full-step features:
 *
 *     x_hat_t = W_i H^T = sum_{j=1..H} W_j x_{f=-j}                           (Eq. 13)
 *
 * The weights W depend only on the timestep differences t - s_j and the hyper-parameters
 * (the "online decoupling" of Sec. 1 and the Diff Key of Eq. 7), so they are solved on
 * the host in fp64 and memoised; the weight application streams every cached byte once
 * through one persistent CUDA kernel.
 *
 * Conventions shared by every call:
 *  - Node j = 1 (C index 0) is the most recent cached feature x_{f=-1}; nodes are listed
 *    newest first everywhere (Sec. 3.2, "Get Key").
 *  - "Layer" is one cached tensor (a block output, or the stepwise feature of Eq. 5),
 *    treated as a flat contiguous vector of `numel` elements.
 *  - Device pointers are plain CUDA device addresses on the device that was current when
 *    the cache was created.  Every device pointer passed in must be 16-byte aligned
 *    (BC_ERR_ALIGNMENT otherwise) and must hold the stated number of elements (the
 *    library cannot check sizes of foreign allocations).
 *  - `stream` is a cudaStream_t passed as void* (NULL = the legacy default stream).  All
 *    device work is enqueued on it asynchronously; errors are reported by return value
 *    only, and no call blocks on the device except bc_cache_create/destroy and
 *    bc_cache_check (and a forecast or push over more than 1016 layers with a new layer
 *    table while four earlier uploads are still queued; see bc_forecast).
 *  - CUDA graphs: while `stream` is being captured, pushes, commits, forecasts (all
 *    variants) and the probe drift enqueue kernels only (no allocation, copy or
 *    synchronisation), so they may be called during capture (outside capture, a forecast or
 *    push over more than 1016 layers may also copy its layer table to the device).  The
 *    graph holds the slot addresses, weights and update coefficients chosen when each call
 *    was made; replaying it repeats that device work and does not move the handle's host
 *    state (ring head, node times, statistics).  The first forecast of each kind on a
 *    device also queries and sets per-device kernel attributes; run the loop once
 *    uncaptured before capturing it.
 *  - Host-side cache state (ring head, node times) changes when the call is made, so
 *    pushes and forecasts on one handle must be issued from one thread, in order, on one
 *    stream (or with the caller's own synchronisation between a push and the calls that
 *    read its slot).  The library orders only its own layer tables across streams.
 *  - No exception crosses the ABI and device code never traps.  The pipeline forecast
 *    kernel and the large drift and push kernels wait on their own shared-memory
 *    pipelines (TMA bulk copies completing on mbarriers); every such wait gives up after
 *    about one second, records the failure in the handle's device status word and
 *    returns, so the device never hangs: bc_cache_check reports it.
 */
#ifndef BARYCACHE_H
#define BARYCACHE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Largest history length H (the paper ablates H = 2, 3, 4: Sec. 4.4). */
#define BC_MAX_K 4

typedef enum {
    BC_OK = 0,
    BC_ERR_INVALID_ARG = 1,        /* bad size, count, dtype, mode, null pointer, overlap */
    BC_ERR_ALIGNMENT = 2,          /* a device pointer is not 16-byte aligned */
    BC_ERR_OOM = 3,                /* device allocation failed (cache arena) */
    BC_ERR_CUDA = 4,               /* a CUDA runtime call failed; see bc_last_error() */
    BC_ERR_NOT_READY = 5,          /* forecast before any feature was pushed */
    BC_ERR_DUPLICATE_NODE = 6,     /* pushed t equals a timestep already in the window */
    BC_ERR_DEGENERATE_WEIGHTS = 7, /* Eq. 11 normaliser vanishes; run a full step instead */
    BC_ERR_BAD_HANDLE = 8,         /* null, destroyed or foreign handle */
    BC_ERR_DEVICE_TIMEOUT = 9      /* a forecast's pipeline wait ran out (bc_cache_check) */
} bc_status;

typedef enum { BC_DTYPE_F32 = 0, BC_DTYPE_BF16 = 1 } bc_dtype;

/* Weight construction.
 *  BC_MODE_EXACT: the polynomial extrapolant through the live nodes, in barycentric form:
 *      c_j = (w_j / (t - s_j)) / sum_k (w_k / (t - s_k)),  w_j = 1 / prod_{k!=j} (s_j - s_k),
 *      and c = e_j exactly when t == s_j (Sec. 1: barycentric interpolation as a
 *      reformulation of polynomial interpolation).
 *  BC_MODE_PAPER: the stabilised weights of Eqs. 8-12 (trapezoid node factors, raw weight
 *      u_j = c_j (-1)^j / (t - s_j), clip to [-C, C], signed decay power with eta, and the
 *      blend lambda towards x_{f=-1}). */
typedef enum { BC_MODE_EXACT = 0, BC_MODE_PAPER = 1 } bc_mode;

typedef struct {
    int32_t mode;   /* bc_mode */
    double delta;   /* decay power of Eq. 11; <= 0 selects delta_H by the live window size
                       H: 1.0 (H <= 2), 0.95 (H = 3), 0.7 (H = 4) (Sec. 3.2, under Eq. 10) */
    double lambda;  /* Eq. 12 blend in [0, 1]: W = (1 - lambda) alpha + lambda e_1 */
    double clip_C;  /* Eq. 10 clip, > 0 (paper: 10) */
    double eta;     /* Eq. 11 offset, >= 0 (paper: 1e-12) */
} bc_params;

typedef struct bc_cache *bc_handle;

/* Kernel selection (bc_cache_set_kernel) for forecasts, probe drifts and push copies.
 * AUTO picks per launch:
 *  - forecast: the shared-memory pipeline (TMA bulk copies into a ring, one CTA per SM:
 *    three stages of 16 KiB per history slot at H <= 3, five of 8 KiB at H = 4) when the
 *    launch has at least 16 of its tiles per SM and its layers average at least 32 tiles,
 *    else the register kernel (each thread holds its history loads in registers; up to two
 *    CTAs per SM; half-size tiles when the launch has fewer than two tiles per SM).  All
 *    forms compute the same bits.
 *  - probe drift: the pipeline form (a five-stage ring of 16 KiB tiles of both tensors, one
 *    CTA per SM) from 16 such tiles per SM on, else register loads.  The two forms group
 *    the partial sums differently, so they agree within rounding, not bit for bit.
 *  - push copy: TMA bulk loads and stores through a three-stage ring (one warp per SM) from
 *    16 tiles of 32 KiB per SM on, else register copies.  Both are byte-exact.
 * REGISTER / PIPELINE pin one form for all three. */
typedef enum { BC_KERNEL_AUTO = 0, BC_KERNEL_REGISTER = 1, BC_KERNEL_PIPELINE = 2 } bc_kernel;

typedef struct {
    int64_t forecasts;       /* successful forecast calls (every bc_forecast* variant) */
    int64_t pushes;          /* successful bc_cache_push / _push_flat / _commit calls */
    int64_t kernel_launches; /* CUDA kernels this handle has launched */
    int64_t memo_hits;       /* Diff Key lookups answered from the memo (Eq. 7) */
    int64_t memo_misses;     /* Diff Key lookups that ran the solver */
    int64_t pipeline_launches; /* of kernel_launches: TMA pipeline kernels (any call) */
    int64_t table_uploads;   /* device layer-table uploads (forecasts and pushes of > 1016
                                layers) */
} bc_stats;

/* ---------------------------------------------------------------- host-only calls */

/* Library ABI version (major * 10000 + minor * 100 + patch). */
int bc_version(void);

/* Static description of a status code.  Never NULL. */
const char *bc_status_string(bc_status s);

/* Detail message of the most recent failing call made by this thread ("" if none).
 * The string stays valid until this thread's next library call. */
const char *bc_last_error(void);

/* Fill `p` with the paper's defaults: PAPER mode, delta by table, lambda 0, C 10,
 * eta 1e-12 (Sec. 3.2; lambda = 0 for C2I/T2I, Sec. 4.1). */
void bc_params_default(bc_params *p);

/* Weight construction (Eqs. 8-12, or the exact barycentric form) for `m` nodes
 * `nodes[0..m-1]` (newest first) and target `t`, in fp64, into c_out[0..m-1].
 * p == NULL uses bc_params_default.  Pure host arithmetic: needs no GPU.
 * Errors: INVALID_ARG (m outside 1..BC_MAX_K, bad params, NaN input),
 * DUPLICATE_NODE (EXACT mode with two equal nodes), DEGENERATE_WEIGHTS. */
bc_status bc_solve(const double *nodes, int m, double t, const bc_params *p, double *c_out);

/* Device bytes a cache of these layers would hold: K slots, each holding every layer at a
 * 256-byte aligned offset (the memory claim of Sec. 1 / Fig. 1: a stepwise cache stores H
 * feature copies, not N x Q).  Needs no GPU. */
bc_status bc_cache_bytes_for(const int64_t *numels, int n_layers, int K, bc_dtype dtype,
                             int64_t *bytes);

/* ------------------------------------------------------------ cache lifecycle */

/* Create the cache context H_t of Eq. 6 for `n_layers` tensors of numels[l] elements of
 * `dtype`, with history length K (1..BC_MAX_K).  Allocates, on the current device, one
 * arena of bc_cache_bytes_for(...) bytes and 16 KiB of reduction scratch for
 * bc_probe_drift plus a status word, and for caches of more than 1016 layers two layer
 * tables (forecast, push) of 32 bytes per layer in device memory, each with four times that
 * of pinned host staging (the only allocations the library makes; freed by
 * bc_cache_destroy).  p == NULL uses the paper's defaults.  Blocks until the allocation is
 * done.  Errors: INVALID_ARG, OOM, CUDA. */
bc_status bc_cache_create(const int64_t *numels, int n_layers, int K, bc_dtype dtype,
                          const bc_params *p, bc_handle *out);

/* Free the arena (synchronises the device first so no enqueued work still reads it). */
bc_status bc_cache_destroy(bc_handle h);

/* Shape of this cache: number of layers, history length K and storage dtype (any of the
 * output pointers may be NULL).  Every per-layer array a call takes or fills has exactly
 * n_layers entries. */
bc_status bc_cache_info(bc_handle h, int *n_layers, int *K, int *dtype);

/* Device bytes held by this cache: the arena, K slots of every layer at 256-byte aligned
 * offsets (not counted: the 16 KiB reduction scratch and status word, the 32-byte-per-layer
 * device layer tables of caches over 1016 layers, and host bookkeeping). */
bc_status bc_cache_bytes(bc_handle h, int64_t *bytes);

/* Replace the weight parameters (clears the weight memo). */
bc_status bc_cache_set_params(bc_handle h, const bc_params *p);

/* Pin the kernel of this handle's forecasts, probe drifts and push copies (bc_kernel;
 * default AUTO). */
bc_status bc_cache_set_kernel(bc_handle h, int kernel);

/* Forget every pushed node (the arena keeps its bytes; nothing is enqueued). */
bc_status bc_cache_reset(bc_handle h);

/* Insert a full-step feature (Eq. 6): the oldest slot is evicted by rotating the ring
 * head, and layer_ptrs[l] (device, numels[l] elements of the cache dtype, 16-byte
 * aligned) is copied into it by one grouped, byte-exact copy kernel on `stream`: with
 * AUTO, TMA bulk copies through a three-stage shared-memory ring (one warp per SM) once the
 * push has at least 16 tiles of 32 KiB per SM, else register loads and stores.  Beyond 1016
 * layers the launch reads its layer table from the handle's device copy, re-uploaded only
 * when the sources differ from the previous push (outside stream capture; while `stream` is
 * captured, one launch per 1016 layers; ordered across streams as for bc_forecast).  The node
 * counts as pushed when the call returns; if the pipeline copy gives up waiting (reported
 * by bc_cache_check) the slot's contents are undefined and the cache should be reset.  `t`
 * is the timestep of this full step.  Errors: INVALID_ARG (null pointer, non-finite t,
 * source overlapping the arena), ALIGNMENT, DUPLICATE_NODE (t equals a node that stays in
 * the window), CUDA. */
bc_status bc_cache_push(bc_handle h, const void *const *layer_ptrs, double t, void *stream);

/* Zero-copy push, part 1: the device addresses (one per layer) of the slot the next push
 * will fill.  The caller (e.g. the DiT writing its block outputs) writes the new feature
 * there, then calls bc_cache_commit.  When the window is full this slot still holds the
 * oldest node, so no forecast may be enqueued between the first write and the commit. */
bc_status bc_cache_next_slot_ptrs(bc_handle h, void **out_ptrs);

/* Zero-copy push, part 2: make the slot returned by bc_cache_next_slot_ptrs the newest
 * node, with timestep t.  No device work.  Errors as bc_cache_push. */
bc_status bc_cache_commit(bc_handle h, double t);

/* Live node timesteps, newest first, into nodes_out[0..*m_out-1] (capacity BC_MAX_K). */
bc_status bc_cache_nodes(bc_handle h, double *nodes_out, int *m_out);

/* Device addresses of node j's stored tensors (j = 0 is x_{f=-1}); j < live count. */
bc_status bc_cache_slot_ptrs(bc_handle h, int j, void **out_ptrs);

/* The weights a forecast at t_new would use (fp64, before rounding to fp32), newest
 * first, m_out = number of live nodes used.  Goes through the Diff Key memo. */
bc_status bc_coefficients(bc_handle h, double t_new, double *c_out, int *m_out);

/* ------------------------------------------------------------ the forecast (Eq. 13) */

/* Skipped-step forecast: for every layer l with out_ptrs[l] != NULL,
 *     out_l[e] = sum_{j=1..m} W_j * F_{l,j}[e],   m = min(pushed, K),
 * with W from the solver (memoised by Diff Key, rounded to fp32), fp32 accumulation in
 * node order j = 1..m, and the result stored as `out_dtype` (bf16: round to nearest even).
 * The fp32 weights are divided by a power of two s >= sum_j |W_j| and the sum multiplied by s
 * at the end: the same bits wherever the plain fp32 sum neither overflows nor goes
 * subnormal, and finite inputs never overflow in a partial sum.  NaN and +-Inf in the history
 * propagate by IEEE rules (a NaN stays NaN; W_j * Inf is an infinity of W_j's sign).
 * One persistent grouped kernel launch covers every selected layer.  Beyond 1016 selected
 * layers the launch reads its layer table from the handle's device copy, which is
 * re-uploaded (one cudaMemcpyAsync on `stream`, from pinned memory) only when the outputs
 * differ from the previous such call; the host waits only if four uploads of different
 * tables are still queued ahead of the device.  Such a call first makes `stream` wait
 * (cudaStreamWaitEvent) for the previous launch that read the table, so forecasts of one
 * handle on several streams never see each other's tables (their outputs remain the
 * caller's to keep apart).  While `stream` is being captured into a CUDA graph it issues
 * one launch per 1016 layers instead, so that the graph holds its own tables.
 * Layers with a NULL output are skipped, which also serves to forecast a window of layers.
 * Outputs must not overlap the arena (checked) or each other (not checked: overlapping
 * outputs race).
 * Errors: INVALID_ARG, ALIGNMENT, NOT_READY, DEGENERATE_WEIGHTS, CUDA. */
bc_status bc_forecast(bc_handle h, double t_new, void *const *out_ptrs, bc_dtype out_dtype,
                      void *stream);

/* Forecast fused with one explicit Euler step of the flow-matching sampler (Sec. 4.1:
 * Euler sampling for T2V).  Layer `v_layer` holds the cached model output (velocity):
 *     v_hat[e] = sum_j W_j V_j[e],    x[e] <- x[e] + dt * v_hat[e]   (fp32 math)
 * in the same launch as the forecast of every other layer with a non-NULL out_ptrs[l].
 * x (device, numels[v_layer] elements of x_dtype, updated in place) must not alias any
 * output.  out_ptrs[v_layer] may be NULL (v_hat not stored) or receive v_hat.
 * dt = t_next - t_new (negative when t runs from 1 to 0).  Errors as bc_forecast. */
bc_status bc_forecast_step(bc_handle h, double t_new, double dt, void *const *out_ptrs,
                           bc_dtype out_dtype, int v_layer, void *x, bc_dtype x_dtype,
                           void *stream);

/* Forecast fused with a general sampler update on layer `v_layer` (the cached model output,
 * e.g. the noise prediction eps of Eq. 3 or a flow velocity), in the same launch as the
 * forecast of every other selected layer:
 *     v_hat[e] = sum_j W_j V_j[e],    x[e] <- a x[e] + b v_hat[e] + c z[e]   (fp32 math;
 * b v_hat is formed inside one FMA from the scaled sum, so x stays finite where only v_hat
 * itself would exceed the fp32 range)
 * z (device, numels[v_layer] elements of x_dtype, 16-byte aligned, read only) may be NULL
 * (no noise term).  Coefficients for the DDPM mean of Eq. 3 and for DDIM come from
 * bc_ddpm_coefficients / bc_ddim_coefficients; Euler is a = 1, b = dt, c = 0
 * (bc_forecast_step).  x and z must not overlap each other, an output or the arena.
 * Errors as bc_forecast_step (INVALID_ARG also for non-finite coefficients). */
bc_status bc_forecast_update(bc_handle h, double t_new, double a, double b, double c,
                             void *const *out_ptrs, bc_dtype out_dtype, int v_layer, void *x,
                             bc_dtype x_dtype, const void *z, void *stream);

/* Skipped-step forecast of every layer into one output buffer laid out like a cache slot:
 * layer l's forecast starts at byte offset offsets[l] of bc_cache_layout, in the cache
 * dtype.  One launch whatever the number of layers (the many-tensor blockwise layout of
 * Sec. 4.5, Tables 5-6), with no per-layer table.  `out` (device, 16-byte aligned,
 * offsets[n_layers] bytes) must not overlap the arena.  The padding between layers is
 * written with unspecified values.  Errors as bc_forecast. */
bc_status bc_forecast_flat(bc_handle h, double t_new, void *out, void *stream);

/* Full-step push (Eq. 6) from one device buffer laid out like a cache slot (layer l at byte
 * offset offsets[l] of bc_cache_layout, in the cache dtype, offsets[n_layers] bytes in all,
 * 16-byte aligned): the oldest slot is evicted and the whole buffer, padding included, is
 * copied into it by one byte-exact copy launch, whatever the number of layers, with no
 * per-layer table (the push counterpart of bc_forecast_flat).  Kernel choice, stream
 * semantics and the give-up behaviour as bc_cache_push.  Errors: INVALID_ARG (NULL src,
 * non-finite t, src overlapping the arena), ALIGNMENT, DUPLICATE_NODE, CUDA. */
bc_status bc_cache_push_flat(bc_handle h, const void *src, double t, void *stream);

/* Byte offset of every layer inside a slot (and inside a bc_forecast_flat output), in
 * offsets[0 .. n_layers-1]; offsets[n_layers] = bytes per slot. */
bc_status bc_cache_layout(bc_handle h, int64_t *offsets);

/* ------------------------------------------------------------ sampler coefficients */

/* DDPM reverse step (Sec. 3.1, Eqs. 2-3) as x_{t-1} = a x_t + b eps + c z:
 * a = 1/sqrt(alpha_t), b = -(1 - alpha_t) / (sqrt(alpha_t) sqrt(1 - alpha_bar_t)), and the
 * Eq. 2 standard deviation c = sqrt(beta_t) with beta_t = 1 - alpha_t (the noise scale of
 * Eq. 1).  Needs 0 < alpha_t <= 1, 0 < alpha_bar_t < 1.  Host only. */
bc_status bc_ddpm_coefficients(double alpha_t, double alpha_bar_t, double *a, double *b,
                               double *c);

/* DDIM step (Song, Meng and Ermon, "Denoising Diffusion Implicit Models", ICLR 2021; the
 * paper's C2I/T2I sampler, Sec. 4.1) from alpha_bar_t to alpha_bar_prev with parameter eta
 * (0 = deterministic), as x_prev = a x_t + b eps + c z:
 *   sigma = eta sqrt((1 - ab_prev)/(1 - ab_t)) sqrt(1 - ab_t/ab_prev),
 *   a = sqrt(ab_prev/ab_t), b = sqrt(1 - ab_prev - sigma^2) - sqrt(ab_prev (1 - ab_t)/ab_t),
 *   c = sigma.
 * Needs 0 < ab_t < 1, ab_t <= ab_prev <= 1, eta >= 0 with 1 - ab_prev - sigma^2 >= 0. */
bc_status bc_ddim_coefficients(double alpha_bar_t, double alpha_bar_prev, double eta, double *a,
                               double *b, double *c);

/* ------------------------------------------------------------ schedules (Sec. 3.3, 4.5) */

/* Equal-spaced schedule: is_full[i] = 1 when step i runs the full model, i.e. i < K (the
 * window fills) or i mod interval == 0; 0 when it is a cache forward.  With K = 2 this
 * gives ceil(n/interval) + 1 full steps, the count implied by the FLOPs of Tables 1 and 3.
 * Host only. */
bc_status bc_schedule_equal(int n_steps, int interval, int K, uint8_t *is_full);

/* Adaptive schedule (Sec. 4.5, Table 5): the relative change of a feature probe between
 * consecutive steps is accumulated and a full step is run once the sum reaches
 * `threshold` (the paper's l), after which the sum restarts at 0.  The first K steps are
 * full (the window fills).  Host-only state, one per sampling run. */
typedef struct {
    double threshold;    /* l */
    double accumulated;  /* drift accumulated since the last full step */
    int32_t K;           /* warm-up full steps */
    int32_t steps;       /* decisions taken */
    int32_t full_steps;  /* of which full */
} bc_adaptive;

bc_status bc_adaptive_init(bc_adaptive *s, double threshold, int K);

/* Decide the next step from its probe drift (>= 0; pass 0 when there is no previous
 * probe): *run_full = 1 for a full step, 0 for a cache forward. */
bc_status bc_adaptive_decide(bc_adaptive *s, double drift, int *run_full);

/* The probe drift of the adaptive schedule, on the device:
 *     out[0] = sum_e |cur[e] - prev[e]|,  out[1] = sum_e |prev[e]|,  out[2] = out[0]/out[1]
 * (out[2] = 0 when both sums are 0, +inf when only out[1] is, NaN when either sum is NaN).
 * cur, prev: device, n elements of dtype, 16-byte aligned; out: 3 device doubles.  Two
 * launches on `stream` with a fixed reduction order (bitwise reproducible on one device for
 * a given kernel choice), using the handle's reduction scratch, so calls on one handle must
 * not overlap on the device.  If the pipeline form gives up waiting (see bc_cache_check),
 * out[] reads NaN.  The caller reads out[2] back to drive bc_adaptive_decide.  Errors:
 * INVALID_ARG, ALIGNMENT, CUDA. */
bc_status bc_probe_drift(bc_handle h, const void *cur, const void *prev, int64_t n,
                         bc_dtype dtype, double *out, void *stream);

/* The probe drift of bc_probe_drift without a handle and without any device allocation, for
 * callers that cannot call cudaMalloc or let a library do so on their behalf: code running
 * inside a host framework that owns every device allocation (a serving engine's memory
 * planner, a plugin interface that forbids allocating outside it), or a latency-bound loop
 * that cannot afford the implicit device synchronisation of cudaMalloc/cudaFree.  The paper
 * has no counterpart; it is a deployment variant of bc_probe_drift.
 * The reduction scratch is a 256 KiB array in the library's own device memory, which every
 * device that loads the library holds until the process exits.  Its capacity bounds the
 * input: n may be at most 1 GiB per tensor (2^29 bf16 or 2^28 fp32 elements); larger n is
 * rejected with INVALID_ARG before anything is enqueued.  cur, prev: device, n elements of
 * dtype, 16-byte aligned; out: 3 device doubles, as bc_probe_drift (same sums, within
 * rounding: the partial sums are grouped differently).  The first call on a device looks up
 * the array's device address (cudaGetSymbolAddress, with that device current), and so does
 * the first call after the device's context was re-created (cudaDeviceReset); make that
 * first call before any stream capture.  Every call shares the one array; it keeps the last
 * call's partial sums, none of which a later call reads before rewriting them, so nothing
 * needs clearing, but calls that overlap on the device (on different streams, or from
 * different threads) race.  Errors: INVALID_ARG, ALIGNMENT, CUDA. */
bc_status bc_probe_drift_noalloc(const void *cur, const void *prev, int64_t n, bc_dtype dtype,
                                 double *out, void *stream);

/* Report device-side failures of this handle's forecast, drift and push launches since the
 * last check: BC_ERR_DEVICE_TIMEOUT if any launch gave up waiting for its shared-memory pipeline
 * (its outputs may then be incomplete), else BC_OK.  Waits for all work on the device, reads and
 * clears the handle's device status word.  Errors: BAD_HANDLE, CUDA, DEVICE_TIMEOUT. */
bc_status bc_cache_check(bc_handle h);

/* Test hook for failure detection (no production use): what = 1 makes the next forecast
 * launch of this handle run the pipeline kernel and leave the first stage of
 * every CTA's pipeline unarmed, so that its bounded wait runs out (about one second) and the
 * launch returns early with the status word set, which bc_cache_check then reports;
 * what = 2 does the same to the next probe drift of at least one 16 KiB tile (its out[]
 * then reads NaN); what = 3 to the next push copy (bc_cache_push or bc_cache_push_flat;
 * the pushed slot is then undefined);
 * what = 0 cancels a pending injection.  Nothing is faulted: the copies
 * that were issued complete and are drained. */
bc_status bc_cache_inject_fault(bc_handle h, int what);

/* Counters of this handle (see bc_stats). */
bc_status bc_cache_stats(bc_handle h, bc_stats *out);

#ifdef __cplusplus
}
#endif

#endif /* BARYCACHE_H */
