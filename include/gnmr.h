/*
 * gnmr.h -- C ABI of libgnmr, the GB300 (sm_103a) implementation of the GNMR
 * per-step monitor: per-unit gradient L2 norms, the online GNMR and
 * Delta-GNMR statistics, and the budgeted choice of the units that move to
 * the higher-fidelity recovery path.
 *
 * Paper: "GNMR: Runtime Stability Control for Low-Precision Large Language
 * Model Training".  Definitions implemented here:
 *   Sec. 2, Eq. local_gradient   n_{b,t} = ||g_{b,t}||_2 per monitored unit b
 *   Sec. 3.1-3.2, Algorithm 1    GNMR, Delta-GNMR, historical mean A, queue Q
 *   Sec. 3.3, Algorithm 2        R = max{GNMR/alpha_t, Delta-GNMR/beta_t},
 *                                C_t = {R > 1} U {Lock > 0}, A_t = Top_maxO,
 *                                Lock bookkeeping
 *   Sec. 3.4                     recoverable vs monitored units, maxO as a
 *                                hard cap, two-stage thresholds
 *
 * Conventions shared by every call:
 *   - Every call returns a gnmr_status; GNMR_OK is 0.  A call that fails its
 *     argument or layout checks returns before anything is enqueued and
 *     leaves the handle's state (step counter included) unchanged.
 *   - Pointers named d_* are CUDA device pointers on the handle's device;
 *     every other pointer is host memory.
 *   - The library owns its state and scratch: one device allocation made by
 *     gnmr_create and freed by gnmr_destroy.  The caller owns the gradient
 *     arena, the mask and the statistics buffers.
 *   - Work is enqueued on the caller's stream (a cudaStream_t passed as
 *     void*, NULL = the legacy default stream).  gnmr_step never blocks the
 *     host; its outputs are valid once that stream reaches the step.
 *   - A handle is not thread-safe: one host thread and one stream at a time.
 *   - The calls save and restore the caller's current CUDA device.
 */
#ifndef GNMR_H
#define GNMR_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum gnmr_status {
    GNMR_OK = 0,
    GNMR_ERR_INVALID_ARG = 1, /* bad pointer, size, threshold or config value */
    GNMR_ERR_LAYOUT = 2,      /* unit layout does not fit the arena given */
    GNMR_ERR_CUDA = 3,        /* a CUDA call failed; the handle is then only good for destroy */
    GNMR_ERR_OOM = 4,         /* host or device allocation failed in gnmr_create */
    GNMR_ERR_STATE = 5        /* handle unusable after an earlier GNMR_ERR_CUDA */
} gnmr_status;

typedef enum gnmr_dtype {
    GNMR_DTYPE_F32 = 0,       /* IEEE binary32 gradients */
    GNMR_DTYPE_BF16 = 1       /* bfloat16 gradients */
} gnmr_dtype;

/* Controller configuration (Sec. 3.3-3.4).  gnmr_config_defaults fills it
 * with the values listed per field. */
typedef struct gnmr_config {
    int32_t num_units;            /* |B|, monitored units, >= 1 (no default) */
    const int64_t *offsets;       /* host [num_units] (or [num_segments]): first element in the arena, >= 0 */
    const int64_t *lengths;       /* host, same count: elements, >= 0 (0 = empty, norm 0) */
    const uint8_t *recoverable;   /* host [num_units], nonzero = b in B_rec; NULL = every unit recoverable */
    int32_t dtype;                /* gnmr_dtype of the arena; default GNMR_DTYPE_BF16 */
    int32_t window;               /* delta, Delta-GNMR window, >= 1; default 8 */
    int32_t max_o;                /* maxO, hard cap on |A_t|, >= 0; default 4 */
    int32_t lock_len;             /* T_lock, >= 0; default 1 */
    double alpha_init;            /* alpha_t for t <= warmup_steps, > 0; default 1.5 */
    double alpha_main;            /* alpha_t for t > warmup_steps, > 0; default 1.1 */
    double beta_init;             /* beta_t for t <= warmup_steps, > 0; default 1.5 */
    double beta_main;             /* beta_t for t > warmup_steps, > 0; default 1.5 */
    int64_t warmup_steps;         /* length of the first threshold stage, >= 0; default 0 */
    double eps;                   /* epsilon of Algorithm 1, >= 0; default 1e-8 */
    int32_t device;               /* CUDA device ordinal; default 0 */
    /* Multi-segment units (Sec. 3.4: a whole transformer block as one
     * recoverable unit, all its operators sharing one decision).  0 (default):
     * unit b is the single segment offsets[b], lengths[b].  > 0: offsets and
     * lengths describe num_segments segments and segment_unit[s] in
     * [0, num_units) names the unit each belongs to; n_b is the L2 norm over
     * all of b's segments (a unit with none has n_b = 0).  Segments may come in
     * any order; a unit's segments are summed in the order given. */
    int32_t num_segments;
    const int32_t *segment_unit;  /* host [num_segments] when num_segments > 0, else ignored */
    /* Policy variants (gnmr_policy; see there).  Defaults: ACTIVE_CAP, 0, 0, 0.25. */
    int32_t policy;
    int64_t forced_recovery_steps; /* steps t <= this: every recoverable unit on the recovery path */
    int64_t static_warmup_steps;   /* GNMR_POLICY_STATIC_TOP: warm-up length */
    double static_fraction;        /* GNMR_POLICY_STATIC_TOP: fraction of B_rec fixed, in [0, 1] */
    /* Extra saved-activation cost c_b of recovering unit b (Eq.
     * generic-memory-bound), host [num_units], copied; NULL = no Delta M_t. */
    const double *unit_cost;
    /* Shape of the kernel's streaming loop (gnmr_loop_shape).  The shapes
     * split the arena into different runs, so norms agree within rounding,
     * not bitwise; each shape is bitwise reproducible call to call (the
     * large-unit shape hands its runs to warps dynamically, but a run's
     * partial sum has a fixed slot and a unit's slots are added in order).
     * Default GNMR_LOOP_AUTO. */
    int32_t loop_shape;
} gnmr_config;

/* Streaming-loop shapes of the step kernel.
 *   GNMR_LOOP_AUTO: GNMR_LOOP_LARGE_UNITS when the mean unit holds at least
 *     1 MiB of gradient, else GNMR_LOOP_SMALL_UNITS.
 *   GNMR_LOOP_SMALL_UNITS: fewer loads in flight per warp, more resident
 *     warps per SM (suits many small units, whose per-unit work overlaps the
 *     stream of other warps).
 *   GNMR_LOOP_LARGE_UNITS: twice the loads in flight per warp, half the
 *     resident warps (suits long streams). */
typedef enum gnmr_loop_shape {
    GNMR_LOOP_AUTO = 0,
    GNMR_LOOP_SMALL_UNITS = 1,
    GNMR_LOOP_LARGE_UNITS = 2
} gnmr_loop_shape;

/* Recovery policies.
 *   GNMR_POLICY_ACTIVE_CAP (default): Algorithm 2, |A_t| <= maxO.
 *   GNMR_POLICY_ADMISSION_CAP: only newly admitted units are capped (the
 *     paper's Remark on the maxO budget): candidates that were on the
 *     recovery path at t - 1 stay; of the other candidates at most maxO, those
 *     with the largest R (ties: lower index), are admitted.  |A_t| can exceed
 *     maxO and is what counts[1] reports.
 *   GNMR_POLICY_STATIC_TOP: the ADAPT-style static baseline (App. E.4): for
 *     t <= static_warmup_steps every recoverable unit is on the recovery path
 *     and its GNMR is summed; at t = static_warmup_steps + 1 the
 *     ceil(static_fraction * |B_rec|) units with the largest sum (ties: lower
 *     index) are fixed on the recovery path for good.
 * Independently, forced_recovery_steps (App. E.7) puts every recoverable
 * unit on the recovery path for t <= forced_recovery_steps, with no candidate
 * pool (statistics still update, locks are left as they are). */
typedef enum gnmr_policy {
    GNMR_POLICY_ACTIVE_CAP = 0,
    GNMR_POLICY_ADMISSION_CAP = 1,
    GNMR_POLICY_STATIC_TOP = 2
} gnmr_policy;

/* Optional per-step statistics: caller-owned DEVICE buffers.  Any pointer
 * may be NULL, and the whole struct may be NULL. */
typedef struct gnmr_stats {
    double *norm;     /* [num_units] n_{b,t} */
    double *gnmr;     /* [num_units] GNMR_{b,t} */
    double *dgnmr;    /* [num_units] Delta-GNMR_{b,t} */
    double *risk;     /* [num_units] R_{b,t} (also reported for non-recoverable units) */
    int32_t *lock;    /* [num_units] Lock_b after the step */
    int32_t *counts;  /* [2]: |C_t|, |A_t| (under STATIC_TOP: the ranked pool, the fixed set) */
    double *delta_mem;/* [1]: Delta M_t = sum of c_b over A_t (needs unit_cost) */
} gnmr_stats;

/* Launch geometry and memory of a handle, for reporting. */
typedef struct gnmr_info {
    int32_t num_units;
    int32_t dtype;
    int32_t device;
    int32_t num_ctas;          /* CTAs per gnmr_step launch */
    int32_t threads_per_cta;
    int32_t num_warps;         /* warps with a work run */
    int64_t num_partials;      /* per-(run, unit) partial sums */
    int64_t device_bytes;      /* library-owned device memory */
    int64_t arena_elems_min;   /* max over units of offset + length */
    int64_t steps;             /* gnmr_step calls enqueued so far */
    int32_t loop_shape;        /* gnmr_loop_shape in use (never GNMR_LOOP_AUTO) */
    int32_t num_runs;          /* work runs: one per warp with the small-unit loop;
                                  about 16 per warp with the large-unit loop, where
                                  each warp starts on its own and then takes the
                                  next untaken one */
} gnmr_info;

typedef struct gnmr_handle gnmr_handle;

/* Fills *cfg with the defaults documented in gnmr_config; num_units,
 * offsets, lengths and recoverable are set to 0 / NULL.  cfg may not be NULL
 * (the call then does nothing). */
void gnmr_config_defaults(gnmr_config *cfg);

/* Validates cfg, copies the unit layout and recoverable flags (the caller may
 * free them afterwards), plans the work partition for the device, allocates
 * and zeroes the per-unit state (A_b, Q_b, k_b, Lock_b) and scratch, and
 * returns a handle in *out.  This is the only call that allocates or blocks.
 * Errors: GNMR_ERR_INVALID_ARG (NULL cfg/out/offsets/lengths, a field out of
 * range, offset + length overflowing), GNMR_ERR_CUDA (device not usable),
 * GNMR_ERR_OOM.  On error *out is set to NULL; gnmr_last_error(NULL) gives
 * the detail. */
gnmr_status gnmr_create(const gnmr_config *cfg, gnmr_handle **out);

/* One training step t = (steps so far) + 1, one kernel launch on `stream`:
 *   1. n_b = ||g_b||_2 for every unit b over the arena (Eq. local_gradient);
 *   2. Algorithm 1 for every unit (k_b plays the role of t: the number of
 *      steps at which b was observed);
 *   3. R_b = max{GNMR/alpha_t, Delta-GNMR/beta_t} (Sec. 3.3), with alpha_t,
 *      beta_t from the two-stage schedule or gnmr_set_thresholds;
 *   4. C_t = {b in B_rec : R_b > 1 or Lock_b > 0};
 *      A_t = the min(maxO, |C_t|) members of C_t with the largest R, ties
 *      broken by the lower unit index (Algorithm 2);
 *   5. Lock_b = T_lock if b in A_t and R_b > 1; max(Lock_b - 1, 0) if b in
 *      A_t and R_b <= 1; 0 otherwise; d_mask[b] = 1 iff b in A_t.
 * A unit whose norm is NaN or Inf gets GNMR = Delta-GNMR = R = +Inf and its
 * A_b, Q_b and k_b are left as they were.
 * Arguments:
 *   d_arena      device-accessible, the flat gradient arena of the
 *                configured dtype, aligned to its element size; read only.
 *                Device memory, or pinned host memory (cudaHostAlloc, or
 *                cudaHostRegister'ed; under unified addressing its host
 *                address is its device address): a host arena is read in
 *                place over the host link, with no staging copy and no
 *                device memory for the gradients; results are bitwise the
 *                same.  May be NULL only if every unit is empty.
 *   arena_elems  elements in d_arena; must be >= max(offset + length)
 *                (else GNMR_ERR_LAYOUT).
 *   stream       cudaStream_t as void*; NULL = legacy default stream.
 *   d_mask       device uint8 [num_units], written (1 = recovery path).
 *   stats        optional statistics outputs (see gnmr_stats), or NULL.
 * The arena must not change until the stream has passed the step.  The
 * kernel is launched as a programmatic dependent of the work before it on
 * the stream: it may be scheduled early, but it waits before its first
 * memory access until that work has completed and its writes are visible,
 * so stream order holds as for a plain launch.  Errors:
 * GNMR_ERR_INVALID_ARG, GNMR_ERR_LAYOUT, GNMR_ERR_STATE, GNMR_ERR_CUDA (the
 * launch failed). */
gnmr_status gnmr_step(gnmr_handle *h, const void *d_arena, int64_t arena_elems,
                      void *stream, uint8_t *d_mask, const gnmr_stats *stats);

/* Sharded step, first half: this rank's per-unit sums of squares.
 *
 * With ZeRO-style sharded data parallelism each rank holds a slice of every
 * unit's gradient, and n_b = ||g_b||_2 needs the sum of the slices' sums of
 * squares (Eq. local_gradient).  The handle is created with the rank's local
 * layout (a unit with no elements on this rank has length 0).  This call
 * reads the local arena like gnmr_step but only writes
 * d_sumsq[b] = sum of g_i^2 over unit b's local elements (device fp64
 * [num_units]); it changes no controller state.  The caller then sums d_sumsq
 * across ranks (e.g. an all-reduce) and calls gnmr_finish on every rank:
 * identical sums give identical masks everywhere.  Arguments and errors as
 * gnmr_step (d_sumsq replaces d_mask).  Launched as gnmr_step is (a
 * programmatic dependent that waits for the preceding work first). */
gnmr_status gnmr_step_partials(gnmr_handle *h, const void *d_arena, int64_t arena_elems,
                               void *stream, double *d_sumsq);

/* Sharded step, second half: one controller step (Algorithms 1 and 2, as in
 * gnmr_step from step 2 on) on given per-unit sums of squares: n_b =
 * sqrt(d_sumsq[b]).  d_sumsq: device fp64 [num_units], read only.  d_mask and
 * stats as in gnmr_step.  Advances the step counter.  Launched as gnmr_step
 * is.  Errors: GNMR_ERR_INVALID_ARG, GNMR_ERR_STATE, GNMR_ERR_CUDA. */
gnmr_status gnmr_finish(gnmr_handle *h, const double *d_sumsq, void *stream, uint8_t *d_mask,
                        const gnmr_stats *stats);

/* Checkpoint: copies the controller state (step counter t, and per unit A_b,
 * k_b, Lock_b, the active flag, the static policy's GNMR sum and the GNMR
 * window Q_b) into host_buf as a self-describing blob ("GNMR", version 2,
 * num_units, window, t, then the per-unit records and windows;
 * little-endian).  *state_bytes (if not NULL) receives the blob size;
 * with host_buf == NULL nothing else happens.  Waits for `stream` (work
 * enqueued on it before the call is included), then returns.  Errors:
 * GNMR_ERR_INVALID_ARG (buf_bytes too small), GNMR_ERR_STATE, GNMR_ERR_CUDA. */
gnmr_status gnmr_get_state(gnmr_handle *h, void *stream, void *host_buf, int64_t buf_bytes,
                           int64_t *state_bytes);

/* Resume: loads a blob written by gnmr_get_state for the same num_units and
 * window into the handle (on `stream`, waited for before returning), so the
 * following steps continue the saved trace exactly.  Errors:
 * GNMR_ERR_INVALID_ARG (NULL, short, foreign or mismatched blob, or a record
 * out of range; the handle is unchanged), GNMR_ERR_STATE, GNMR_ERR_CUDA. */
gnmr_status gnmr_set_state(gnmr_handle *h, void *stream, const void *host_buf, int64_t buf_bytes);

/* Overrides alpha_t and beta_t for the following steps ("scheduled
 * relaxation", Sec. 3.4).  NaN for either value returns it to the two-stage
 * schedule.  Other values must be finite and > 0 (else
 * GNMR_ERR_INVALID_ARG). */
gnmr_status gnmr_set_thresholds(gnmr_handle *h, double alpha, double beta);

/* Reports the launch geometry and memory of the handle into *info. */
gnmr_status gnmr_get_info(const gnmr_handle *h, gnmr_info *info);

/* Waits for work in flight on the handle's device, frees everything the handle owns and the
 * handle itself.  NULL is accepted (GNMR_OK). */
gnmr_status gnmr_destroy(gnmr_handle *h);

/* Static text for a status code. */
const char *gnmr_status_string(gnmr_status s);

/* Detail of the last failure on h; with h == NULL, of the last failed call
 * without a handle (gnmr_create, the actuator calls, gnmr_unit_norms_static)
 * on the calling thread.  Valid until the next call on h (or
 * create on this thread); never NULL. */
const char *gnmr_last_error(const gnmr_handle *h);

/* Host-only query of the work partition that gnmr_create plans for the
 * small-unit loop shape (max_warps = the resident warps): the concatenation
 * of all units (an empty unit counts as one element of work) is cut into at
 * most max_warps contiguous runs of about equal cost (element bytes plus a
 * fixed per-unit cost), one run per warp.  (The large-unit shape cuts the
 * same way into about 16 runs per warp, see gnmr_info.num_runs.)  Outputs,
 * caller-allocated: run_unit / run_pos [max_warps + 1] (run w covers
 * (run_unit[w], run_pos[w]) up to, not including, (run_unit[w+1],
 * run_pos[w+1])), first_warp / num_parts [num_units] (the warps touching
 * unit b are first_warp[b] .. first_warp[b] + num_parts[b] - 1).  *num_warps
 * receives the number of runs.  No CUDA call is made.  Errors:
 * GNMR_ERR_INVALID_ARG. */
gnmr_status gnmr_plan_partition(int32_t num_units, const int64_t *lengths, int32_t dtype,
                                int32_t max_warps, int32_t *num_warps, int32_t *run_unit,
                                int64_t *run_pos, int32_t *first_warp, int32_t *num_parts);

/* ---- Recovery actuator (App. E.2; the stress bench of Sec. 5.1) --------
 * The mask decides, per unit, which path the unit's saved activations take:
 * the low-cost format or the higher-fidelity recovery format.  The actuator
 * fake-quantizes each unit's activations token by token: for every row,
 * amax = max |x|, inv = fmax / amax, scale = amax / fmax, and
 * y = round(x * inv) * scale, where round() gives the nearest value
 * representable in the format (ties to the even code, saturating at fmax).
 * All of this is fp32 arithmetic.  Rows whose amax is 0 or that hold a NaN or
 * Inf are copied unchanged. */
typedef enum gnmr_fq_format {
    GNMR_FQ_NONE = 0,   /* copy (no quantization) */
    GNMR_FQ_E2M1 = 1,   /* 4-bit: 2 exponent bits (bias 1), 1 mantissa bit, max 6 */
    GNMR_FQ_E3M2 = 2,   /* 6-bit: bias 3, max 28 */
    GNMR_FQ_E4M3 = 3,   /* 8-bit: bias 7, max 448 */
    GNMR_FQ_E5M2 = 4    /* 8-bit: bias 15, max 57344 */
} gnmr_fq_format;

typedef struct gnmr_actuator gnmr_actuator;

/* Activation layout: unit b's activations are a row-major [rows[b] x
 * cols[b]] block (one row per token) starting at element offsets[b] of a flat
 * buffer of `dtype` (host arrays, copied).  Errors: GNMR_ERR_INVALID_ARG,
 * GNMR_ERR_CUDA, GNMR_ERR_OOM; detail via gnmr_last_error(NULL). */
gnmr_status gnmr_actuator_create(int32_t num_units, const int64_t *offsets, const int64_t *rows,
                                 const int64_t *cols, int32_t dtype, int32_t device,
                                 gnmr_actuator **out);

/* Fake-quantizes every unit's activations from d_in into d_out (device, same
 * layout; d_out == d_in works in place) on `stream`: unit b uses
 * recovery_format if d_mask[b] != 0, else lowcost_format (d_mask: device
 * uint8 [num_units] as written by gnmr_step, or NULL = low-cost for all).
 * arena_elems bounds both buffers.  Errors: GNMR_ERR_INVALID_ARG,
 * GNMR_ERR_LAYOUT, GNMR_ERR_CUDA. */
gnmr_status gnmr_actuator_apply(gnmr_actuator *a, const void *d_in, void *d_out, int64_t arena_elems,
                                const uint8_t *d_mask, int32_t lowcost_format,
                                int32_t recovery_format, void *stream);

/* Frees the actuator (waits for its device).  NULL is accepted. */
gnmr_status gnmr_actuator_destroy(gnmr_actuator *a);

/* Allocation-free per-unit norms.  The paper has no counterpart: this is a
 * deployment variant of the first stage of gnmr_step.
 *
 * For callers that cannot allocate device memory -- code running inside a
 * framework whose caching allocator already owns the GPU's memory, hooks
 * called in the middle of a training step (where cudaMalloc/cudaFree would
 * synchronise the device), deployments with a footprint fixed at start-up --
 * and therefore cannot hold a gnmr_handle.  Computes n_b = ||g_b||_2 for
 * every unit (the values gnmr_step writes to stats->norm) into d_norms, using
 * as scratch only a device array that lives in the library's static data:
 * about 5.6 MiB, reserved on every GPU that loads the library until the
 * process exits.  No cudaMalloc, cudaFree or other allocating call is made.
 *
 * Arguments: d_arena (device, dtype elements, aligned to the element size;
 * NULL only if every unit is empty), arena_elems, dtype (gnmr_dtype),
 * num_units, offsets / lengths (HOST arrays of num_units elements, copied on
 * the stream before the call returns), d_norms (device fp64 [num_units],
 * written), stream (cudaStream_t as void*, NULL = legacy default stream).
 * Runs on the calling thread's current device.
 *
 * Limit: num_units <= 131072 (any arena size); beyond it
 * GNMR_ERR_INVALID_ARG, with gnmr_last_error(NULL) reading "units > 131072".
 * The arena is read as 64 KiB chunks split into contiguous ranges over the
 * GPU's warps, at the step kernel's streaming rate.  A unit outside [0, arena_elems)
 * gives GNMR_ERR_LAYOUT ("unit off arena"); other details: "dtype unknown",
 * "NULL pointer", "arena misalign", "CUDA failed", "device query" (the
 * current device or its SM count could not be read).  The call makes no host
 * allocation either, on success or failure.
 *
 * The first call on a device looks up the array's device address for that
 * device; make that first call before any stream capture.  The layout tables
 * are uploaded (pageable host->device copies) only when the layout, dtype or
 * device differs from the previous call's; a call repeating the previous
 * layout enqueues one memset and one kernel.  Every call shares the one
 * array and leaves its contents behind (each call clears what must start at
 * zero); calls that overlap on the GPU race on it, so callers must serialise
 * them (one stream, one thread at a time).  Each upload tags the tables with
 * a new generation number and every kernel checks it: a kernel that runs
 * after another call has replaced the tables with a different layout writes
 * NaN for every unit instead of norms of the wrong layout.  The array's
 * address is cached per device for the life of the process: after a
 * cudaDeviceReset this function must not be called again on that device. */
gnmr_status gnmr_unit_norms_static(const void *d_arena, int64_t arena_elems, int32_t dtype,
                                   int32_t num_units, const int64_t *offsets,
                                   const int64_t *lengths, double *d_norms, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* GNMR_H */
