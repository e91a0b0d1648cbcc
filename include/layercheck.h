/*
 * layercheck.h -- C ABI of the GB300 LayerCheck hot path (liblayercheck.so).
 *
 * LayerCheck (adaptive layer-wise checkpointing, §3) persists at every
 * checkpoint opportunity only the layers whose normalized weight drift has
 * reached a threshold, plus any layer that has gone S_max steps without
 * persistence; each persisted layer carries its weights and their Adam
 * moments; recovery assembles, per layer, the latest persisted version.
 *
 * This library runs the per-step path on one GPU:
 *   lc_measure   §3.2 Eq. 1   per-layer normalized update u_l (sm_103a kernel)
 *   lc_select    §3.2 Eq. 2-4 and §3.3 staleness guard (sm_103a kernel)
 *   lc_pack_*    §3.1 full layer state of the selected layers into one
 *                contiguous packed stream, optionally on to pinned host memory
 *   lc_commit_snapshot        reference snapshot <- weights, selected layers
 *   lc_restore   §3.5 / Eq. 8 mixed-timestamp composite back into place
 *
 * Conventions for every call:
 *   - Every entry point returns lc_status; LC_OK is 0.  On any other value
 *     lc_last_error() returns a message (thread-local, valid until the next
 *     call on the same thread).  No call throws or aborts.
 *   - "device" pointers are CUDA device (or managed) memory of the context's
 *     device; "host" pointers are ordinary host memory unless stated.
 *   - The caller owns every tensor it registers (weights, snapshot, Adam
 *     moments) and the CUDA stream it passes to lc_create.  The library
 *     keeps raw pointers: they must stay valid and must not move until
 *     lc_destroy.  The library owns its own tables, staging ring, per-layer
 *     state, pinned result block and the stores it creates.
 *   - Work is enqueued on the context's stream in call order.  The caller
 *     must not modify a registered tensor between lc_measure and the end of
 *     that step's lc_pack_* / lc_commit_snapshot work on the stream (record
 *     an event on the stream and make the training stream wait on it).
 *   - A context is not thread-safe; use one context per thread or lock.
 *   - Call order per context (LC_ERR_STATE otherwise):
 *       lc_register_layout once, then per step
 *       lc_measure -> [all-reduce of lc_layer_sums_device] -> lc_select
 *         -> (lc_pack_device | lc_pack_async) -> lc_commit_snapshot
 *     A step in which lc_select selected nothing may go straight to the next
 *     lc_measure.  lc_restore may be called whenever no step is open.
 */
#ifndef LAYERCHECK_H
#define LAYERCHECK_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    LC_OK = 0,
    LC_ERR_INVALID_ARG = 1,  /* an argument is out of range or inconsistent   */
    LC_ERR_STATE = 2,        /* the call is out of order for this context     */
    LC_ERR_CUDA = 3,         /* a CUDA runtime call or kernel launch failed   */
    LC_ERR_OOM = 4,          /* device or pinned host allocation failed       */
    LC_ERR_CAPACITY = 5,     /* a destination or store is too small           */
    LC_ERR_TIMEOUT = 6,      /* a bounded host wait on the GPU ran out        */
    LC_ERR_NOT_FOUND = 7     /* no persisted version satisfies the request    */
} lc_status;

typedef enum { LC_BF16 = 0, LC_F32 = 1 } lc_dtype;

/* How the reference weights R of Eq. 1 are kept.
 * LC_DRIFT_SNAPSHOT  : R is the layer's weights at its last persistence, so
 *                      u_l is the drift accumulated since then and is used
 *                      directly as the accumulator (Eq. 2 measured end to
 *                      end); lc_commit_snapshot refreshes R for persisted
 *                      layers only.
 * LC_DRIFT_ACCUMULATE: R is W(t-1) (Eq. 1 literally); lc_measure also writes
 *                      R <- W for every layer and Eq. 2 sums u_l over steps. */
typedef enum { LC_DRIFT_SNAPSHOT = 0, LC_DRIFT_ACCUMULATE = 1 } lc_drift_mode;

/* How the kernels move bytes (the results are the same either way).
 * LC_COPY_BULK   : the bulk-copy engine (cp.async.bulk through shared-memory
 *                  rings, one load-issuing thread per CTA) whenever every
 *                  address involved is device memory: the pack, commit and
 *                  restore copies (segments, staging ring and destination),
 *                  the measure's reads of W and R (and its R <- W in
 *                  LC_DRIFT_ACCUMULATE mode), and the fused AdamW step.
 *                  Otherwise as LC_COPY_THREADS (default).
 * LC_COPY_THREADS: every thread loads (and stores) 16-byte vectors. */
typedef enum { LC_COPY_BULK = 0, LC_COPY_THREADS = 1 } lc_copy_engine;

/* Test switches of the bulk engine's bounded waits (they fault and hang
 * nothing).  With one set, each CTA of the kernel named waits for 16 bytes
 * that never arrive: the wait gives up after 1 s, the kernel sets the
 * context's fault word and returns without finishing its work, and from
 * then on lc_select, lc_wait_durable, lc_step_wait and lc_restore fail with
 * LC_ERR_TIMEOUT.
 * Every CTA of the copy kernel reads a device-memory copy of the fault word
 * before its first load and returns at once if it is set, so a copy launch
 * of several waves of CTAs ends soon after its first wave gave up, and later
 * copy launches of the context end at once.
 * LC_DEBUG_BULK_STALL   : the pack / commit / restore copy kernel.
 * LC_DEBUG_MEASURE_STALL: the bulk-load measure kernel and the bulk-load
 *                         fused AdamW step (they share the work partition). */
#define LC_DEBUG_BULK_STALL 1
#define LC_DEBUG_MEASURE_STALL 2

/* One parameter tensor ("segment") of a layer (§2.2: embed_tokens, each
 * transformer block, the final norm and lm_head are the layers; a layer
 * may hold several tensors).
 *   layer      : layer id in [0, nlayers)
 *   w_dtype    : lc_dtype of w and snap
 *   w          : device, numel elements, current weights W_l(t); must be
 *                aligned to its element size (written only by lc_restore)
 *   snap       : device, numel elements of w_dtype, the reference weights R
 *                (written by commit / accumulate mode / restore); may be
 *                NULL in LC_DRIFT_ACCUMULATE mode for a context that measures
 *                only through lc_adamw_step_measure (lc_measure then fails)
 *   exp_avg    : device, numel fp32 Adam first moment, or NULL
 *   exp_avg_sq : device, numel fp32 Adam second moment; NULL iff exp_avg is
 *   numel      : > 0
 * Segments must not overlap one another. */
typedef struct {
    int32_t layer;
    int32_t w_dtype;
    void* w;
    void* snap;
    float* exp_avg;
    float* exp_avg_sq;
    int64_t numel;
} lc_segment;

typedef struct {
    double eps_w;            /* Eq. 1 stabiliser epsilon_w (default 1e-8)        */
    int32_t mode;            /* lc_drift_mode (default LC_DRIFT_SNAPSHOT)         */
    int32_t pack_align;      /* section alignment of the packed layout, a power
                                of two >= 16 (default 256)                        */
    int32_t fuse_commit;     /* 1: lc_pack_* also writes snap <- w for the packed
                                weights, and lc_commit_snapshot launches nothing
                                (default 1)                                       */
    int32_t timeout_ms;      /* bound of every host wait (default 60000)          */
    uint64_t staging_bytes;  /* device staging ring used by lc_pack_async and
                                lc_restore, split in two slots (default 512 MiB) */
    int32_t copy_engine;     /* lc_copy_engine (default LC_COPY_BULK)            */
    int32_t debug_flags;     /* 0, or LC_DEBUG_* switches (tests only)           */
} lc_config;

typedef struct lc_ctx lc_ctx;
typedef struct lc_store lc_store;

/* Outcome of the last lc_select (§3.3 staleness statistics included). */
typedef struct {
    int64_t step;                /* the step passed to lc_measure               */
    int32_t n_selected;          /* layers persisted at this step               */
    int32_t n_nonfinite;         /* layers whose accumulated drift was not finite
                                    (selected; conservative counting)          */
    uint64_t bytes;              /* packed stream size of the selected layers   */
    int64_t max_staleness;       /* max_l (t - t_l) after this step             */
    double weighted_staleness;   /* sum_l n_l (t - t_l) / sum_l n_l after it    */
} lc_select_info;

/* One persisted layer version in a store (the per-layer persistence
 * history of §3.5, "metadata-driven reconstruction"). */
typedef struct {
    int32_t layer;
    int32_t durable;         /* 1 once its device->host copy is known complete */
    int64_t step;            /* t_l of this version                            */
    const void* host_ptr;    /* packed layer block in the store (pinned host)  */
    uint64_t bytes;          /* block size; equals lc_layer_block_bytes(layer) */
} lc_version;

/* Counters of work the context has enqueued (monotone). */
typedef struct {
    int64_t kernel_launches;     /* every kernel this library launched          */
    int64_t measure_launches;
    int64_t select_launches;
    int64_t copy_launches;       /* pack / commit / restore copy kernels        */
    uint64_t d2h_bytes;          /* bytes copied device -> host by the library  */
    uint64_t h2d_bytes;          /* bytes copied host -> device by the library  */
    int64_t bulk_copy_launches;  /* copy launches that ran on the bulk engine   */
    int64_t bulk_measure_launches; /* measure launches on the bulk engine       */
    int64_t measure_pool_units;    /* small ranges that the bulk measure's CTAs
                                      take from a pool after their own (0: the
                                      layout is too small for one)             */
} lc_counters;

/* Fills cfg with the defaults listed in lc_config. */
void lc_config_default(lc_config* cfg);

/* Message of the last failing call on this thread ("" if none). */
const char* lc_last_error(void);

/* Creates a context on CUDA device `device` that enqueues its work on
 * `cuda_stream` (a cudaStream_t; NULL = the legacy default stream).  The
 * stream stays owned by the caller.  cfg may be NULL (defaults).
 * Errors: INVALID_ARG (bad device or config), CUDA, OOM. */
lc_status lc_create(lc_ctx** out, int device, void* cuda_stream, const lc_config* cfg);

/* Waits (bounded) for the context's work and frees everything it owns. */
void lc_destroy(lc_ctx* ctx);

/* Registers the layer -> tensor segment table, once per context (§2.2
 * layer partition; §3.4.1 layer-aligned optimizer state).  segs: host
 * array of nseg entries; every layer in [0, nlayers) needs >= 1 segment.
 * A layer's segments keep their registration order in every sum and in
 * the packed layout.  tau_mult: host array of nlayers finite factors >= 0
 * applied to tau per layer (e.g. 10 for embeddings, §3.4.3), or NULL (1).
 * Resets the accumulators Delta_l = 0 and last-persistence steps t_l = 0:
 * the registered weights and snapshot are the base state of step 0.
 * Errors: INVALID_ARG (layout, pointers not device memory, misaligned
 * element pointers), STATE (already registered), OOM, CUDA. */
lc_status lc_register_layout(lc_ctx* ctx, const lc_segment* segs, int32_t nseg,
                             int32_t nlayers, const double* tau_mult);

/* §3.2 Eq. 1: enqueues the segmented reduction sum|W - R|, sum|R| and the
 * element count per layer (fp32 partial sums of at most 32 terms, combined
 * in fp64 in a fixed order: deterministic for a given layout and device).
 * In LC_DRIFT_ACCUMULATE mode also writes R <- W for every segment.
 * step: the checkpoint opportunity t, strictly greater than the previous
 * step (>= 0 for the first).  Asynchronous.
 * Errors: STATE (not registered, or a step is open), INVALID_ARG, CUDA. */
lc_status lc_measure(lc_ctx* ctx, int64_t step);

/* Device pointer to 3*nlayers fp64 values (D_l, A_l, n_l) per layer, valid
 * after lc_measure in stream order.  A data-parallel caller that shards
 * every layer across ranks all-reduces (sums) this array in place on the
 * context's stream before lc_select, so every rank takes the same
 * decision.  Errors: STATE (not registered). */
lc_status lc_layer_sums_device(lc_ctx* ctx, double** sums_dev);

/* Makes the context keep the per-layer sums in a caller-owned device buffer
 * of 3*nlayers fp64 (8-byte aligned) instead of its own, e.g. a tensor the
 * caller all-reduces with its collective library.  The buffer must stay
 * valid until lc_destroy or the next call.  Errors: STATE (not registered,
 * or a step is open), INVALID_ARG (NULL, misaligned or not device memory). */
lc_status lc_set_layer_sums_buffer(lc_ctx* ctx, double* sums_dev);

/* §3.2 Eq. 2-4 and §3.3: on the device, u_l from the sums, the accumulator
 * update, persist if Delta_l >= tau * tau_mult[l] or t - t_l >= max_staleness
 * or the drift is not finite, then Delta_l <- 0, t_l <- t for the persisted
 * layers; lays out the packed stream (selected layers ascending).  Blocks
 * until the decision is in host memory (bounded by timeout_ms).
 * tau: finite threshold K(t) already scaled by the learning-rate schedule.
 * max_staleness: S_max >= 0 (0 persists every layer every step).
 * mask_out (nlayers bytes, 1 = persist), u_out (nlayers fp64), bytes_out:
 * host, each may be NULL.
 * Errors: STATE (no lc_measure since the last select), INVALID_ARG,
 * TIMEOUT, CUDA. */
lc_status lc_select(lc_ctx* ctx, double tau, int32_t max_staleness,
                    uint8_t* mask_out, double* u_out, uint64_t* bytes_out);

/* Statistics of the last lc_select.  Errors: STATE (none yet). */
lc_status lc_last_select_info(const lc_ctx* ctx, lc_select_info* out);

/* Host array of nlayers: byte offset of each selected layer's block in the
 * packed stream of the last lc_select (0 for unselected layers). */
lc_status lc_last_select_offsets(const lc_ctx* ctx, uint64_t* offsets_out);

/* §3.1 full layer state: gathers the selected layers' weights, exp_avg and
 * exp_avg_sq into dst (device, 16-byte aligned, dst_capacity bytes).
 * Layout: selected layers ascending by id; per layer every segment's W
 * bytes, then every segment's exp_avg, then every exp_avg_sq, each section
 * starting at a multiple of pack_align and zero-padded.  Asynchronous.
 * With fuse_commit also writes snap <- w for those layers.
 * Errors: STATE (no select), INVALID_ARG, CAPACITY (bytes > capacity), CUDA. */
lc_status lc_pack_device(lc_ctx* ctx, void* dst, uint64_t dst_capacity);

/* Same packed stream, through the device staging ring into `store` in
 * pinned host memory (device->host copies on the library's copy stream).
 * Records one pending version per selected layer; they become durable in
 * lc_wait_durable (a step that persisted nothing is durable at once).
 * Asynchronous, except that with a newest-only store it may wait for
 * copies of this step to make room (see lc_store_create).  Errors: STATE (no
 * select, or the store still holds a pending version of a layer it would
 * overwrite; for a newest-only store, any pending version), INVALID_ARG
 * (store built for another layout), CAPACITY, TIMEOUT, CUDA. */
lc_status lc_pack_async(lc_ctx* ctx, lc_store* store);

/* Snapshot mode: enqueues snap <- w for the layers persisted this step
 * (Eq. 4 resets the drift reference with the accumulator); a no-op launch-
 * wise with fuse_commit or in accumulate mode.  Closes the step.
 * Errors: STATE (persisted layers were not packed). */
lc_status lc_commit_snapshot(lc_ctx* ctx);

/* Waits (polling, at most timeout_ms; <= 0 uses the config's) until the
 * device->host copies of `step` issued by lc_pack_async have completed and
 * marks those versions durable ("successfully persisted", §3.1).
 * Errors: NOT_FOUND (no pending pack of that step), TIMEOUT, CUDA. */
lc_status lc_wait_durable(lc_ctx* ctx, int64_t step, int32_t timeout_ms);

/* §3.5 / Eq. 8: for every layer, the durable version in `store` with the
 * largest step <= t_fail; copies those blocks host->device and scatters
 * them into w, exp_avg, exp_avg_sq and snap (snap <- the restored w).  Sets
 * t_l to each version's step and Delta_l = 0.  Blocks until done.
 * layer_steps_out: host, nlayers, the chosen steps (nullable).
 * Errors: NOT_FOUND (some layer has no version <= t_fail), STATE,
 * INVALID_ARG, TIMEOUT, CUDA. */
lc_status lc_restore(lc_ctx* ctx, lc_store* store, int64_t t_fail, int64_t* layer_steps_out);

/* Size of one packed layer block (host-side layout query, §3.1). */
lc_status lc_layer_block_bytes(const lc_ctx* ctx, int32_t layer, uint64_t* out);

/* Library-side work counters of the context. */
lc_status lc_get_counters(const lc_ctx* ctx, lc_counters* out);

/* --- steps without a host round trip ------------------------------------ */

/* One whole step -- measure (Eq. 1), select (Eq. 2-4, §3.3), pack of the
 * persisted layers' full state (§3.1) into dst, snapshot commit -- enqueued
 * on the context's stream with no host synchronization: the pack reads its
 * size from device memory.  dst: device or pinned host memory (16-byte
 * aligned; a pinned host buffer receives the stream directly over the host
 * link), dst_capacity bytes.  If the step's stream would exceed
 * dst_capacity, nothing is persisted and every layer keeps the
 * not-persisted update (its drift stays accumulated); lc_step_wait then
 * returns LC_ERR_CAPACITY.  Up to 4 steps may be in flight; the decision
 * of each is read with lc_step_wait.  Requires snapshots (lc_measure's
 * rules).  Errors: STATE (a step open, 4 in flight, no snapshot),
 * INVALID_ARG, CUDA. */
lc_status lc_step_async(lc_ctx* ctx, int64_t step, double tau, int32_t max_staleness,
                        void* dst, uint64_t dst_capacity);

/* Waits (bounded) for step `step` of lc_step_async or lc_step_graph_launch
 * and returns its decision like lc_select (host arrays nullable); also
 * updates lc_last_select_info / lc_last_select_offsets.
 * Errors: NOT_FOUND (no such step in flight), CAPACITY (the step persisted
 * nothing, see lc_step_async), TIMEOUT, CUDA. */
lc_status lc_step_wait(lc_ctx* ctx, int64_t step, int32_t timeout_ms, uint8_t* mask_out,
                       double* u_out, uint64_t* bytes_out);

/* Captures the sequence of lc_step_async once as a CUDA graph with fixed
 * tau, max_staleness and destination; the step number then comes from a
 * device counter (previous step + 1).  Replaces an earlier graph of this
 * context.  Errors: STATE, INVALID_ARG, CUDA. */
lc_status lc_step_graph_create(lc_ctx* ctx, double tau, int32_t max_staleness, void* dst,
                               uint64_t dst_capacity);

/* Launches the captured step on the context's stream; *step_out (nullable)
 * receives its step number.  The previous graph step must have been read
 * with lc_step_wait.  Errors: STATE (no graph, or its last step not
 * waited for), CUDA. */
lc_status lc_step_graph_launch(lc_ctx* ctx, int64_t* step_out);

/* --- fused optimizer step with the drift read off the update ------------ */

/* Optimizer inputs of one segment, in the registration order of
 * lc_register_layout.  The segment's w must be its fp32 (master) weights and
 * its exp_avg / exp_avg_sq must be set.
 *   grad       : device, numel elements of grad_dtype (LC_BF16 or LC_F32)
 *   model_copy : device, numel bf16 elements that receive the updated
 *                weights rounded to nearest even (e.g. the model's bf16
 *                parameters), or NULL */
typedef struct {
    const void* grad;
    int32_t grad_dtype;
    int32_t reserved;
    void* model_copy;
} lc_optim_segment;

/* AdamW hyperparameters (decoupled weight decay). */
typedef struct {
    double lr, beta1, beta2, eps, weight_decay;
} lc_adamw_hparams;

/* Registers the gradient and model-copy pointers of every segment (§3.4.2:
 * the drift is computed on the optimizer update path).  Requires a layout
 * in LC_DRIFT_ACCUMULATE mode whose segments all have fp32 w and Adam
 * moments.  Errors: STATE (no layout, or snapshot mode), INVALID_ARG. */
lc_status lc_register_optimizer(lc_ctx* ctx, const lc_optim_segment* segs, int32_t nseg);

/* One AdamW step on every registered segment, in place on w, exp_avg and
 * exp_avg_sq (and model_copy), with the Eq. 1 sums of the update taken on
 * the same pass: D_l = sum |w_new - w_old|, A_l = sum |w_old|, so W(t-1) is
 * the weights before this update and no separate scan reads them again.
 * Takes the place of lc_measure for the step (then lc_select accumulates,
 * Eq. 2).  step = t >= 1 is also the bias-correction count.  fp32
 * arithmetic, one rounding per operation in this order: p *= 1 - lr*wd;
 * m = beta1*m + (1-beta1)*g; v = beta2*v + (1-beta2)*(g*g);
 * v_hat = v * (1/(1-beta2^t)); p -= (m * (lr/(1-beta1^t))) / (sqrt(v_hat) + eps);
 * the fp32 constants are formed in binary64 and rounded once.  Asynchronous.
 * Errors: STATE (no optimizer registered, or a step is open), INVALID_ARG. */
lc_status lc_adamw_step_measure(lc_ctx* ctx, int64_t step, const lc_adamw_hparams* hp);

/* --- copy trace (measurement of the staged host copies) ---------------- */

/* What a traced span timed.  lc_pack_async stages its stream through the
 * device staging ring in chunks: for each chunk a GATHER span on the
 * context's stream (the pack kernel into a staging slot) and a D2H span on
 * the library's copy stream (the device->host copies of that slot into the
 * store).  lc_restore does the reverse: an H2D span on the copy stream, then
 * a SCATTER span on the context's stream. */
#define LC_SPAN_GATHER 0
#define LC_SPAN_D2H 1
#define LC_SPAN_H2D 2
#define LC_SPAN_SCATTER 3

typedef struct {
    int32_t kind;       /* LC_SPAN_*                                            */
    int32_t chunk;      /* chunk index within its lc_pack_async / lc_restore    */
    int64_t step;       /* the packed step, or t_fail of the restore            */
    uint64_t bytes;     /* bytes of the packed stream the chunk covers          */
    double start_ms;    /* ms after the first recorded span started (NaN if the */
    double end_ms;      /* span could not be timed)                             */
} lc_copy_span;

/* Starts (enable != 0) or stops recording spans; either way the previous
 * record is cleared.  A span's start event is recorded on its stream just
 * before its work and its end event just after, so end - start is the work
 * itself, and the gap between consecutive spans of one stream is time that
 * stream spent waiting (for the other stream or for its own earlier work).
 * Costs two CUDA events per span; at most 65536 spans are kept, later ones
 * are counted as dropped.  Errors: INVALID_ARG. */
lc_status lc_copy_trace_enable(lc_ctx* ctx, int32_t enable);

/* Waits (bounded by the config's timeout_ms) for the recorded spans and
 * copies up to `cap` of them, in record order, into `out` (host).  *n_out
 * (nullable): spans recorded; *dropped_out (nullable): spans not kept.  Does
 * not clear the record.  Errors: INVALID_ARG, TIMEOUT, CUDA. */
lc_status lc_copy_trace_read(lc_ctx* ctx, lc_copy_span* out, int64_t cap, int64_t* n_out,
                             int64_t* dropped_out);

/* --- persisted-version store (pinned host memory) ---------------------- */

/* Creates a store for the layout registered in ctx.
 * versions_per_layer = 0: an append-only log of every version in one
 *   pinned arena of capacity_bytes (every restore point stays available
 *   until lc_store_clear).
 * versions_per_layer = 1: newest-only.  An arena of capacity_bytes holds
 *   each layer's newest durable version.  Layers whose blocks have the same
 *   size share a class of slots: the class's layers' slots, one spare, and
 *   further spares as capacity_bytes allows (4096-byte aligned).  A new
 *   version goes into a free slot of its class, and the layer's previous
 *   version frees its slot only once the new one is durable, so a crash
 *   during a copy still leaves the previous version.  Durability is per
 *   layer: a version counts as durable as soon as its own copy has completed.
 *   When a class has no free slot, lc_pack_async waits (host side, bounded by
 *   timeout_ms) for the copy of the step's earliest layer of that class not
 *   yet seen complete, whose previous version's slot then serves; so every
 *   step fits, whatever it persists, in every layer's block plus one block of
 *   each distinct size (the minimum capacity_bytes accepted).  The placement
 *   is decided before anything is enqueued: LC_ERR_CAPACITY (possible only
 *   after exclusions) leaves the store untouched.  lc_pack_async needs every
 *   earlier version durable (lc_wait_durable).  Only the newest restore point
 *   of each layer is available.
 * versions_per_layer = V >= 2: each layer owns V block slots and keeps its
 *   V newest versions; capacity_bytes is ignored.  Restore points older
 *   than a layer's oldest kept version are no longer available.
 * The store is pinned with cudaHostAlloc and owned by the library.
 * Errors: INVALID_ARG, STATE (ctx not registered), OOM. */
lc_status lc_store_create(lc_store** out, const lc_ctx* ctx, uint64_t capacity_bytes,
                          int32_t versions_per_layer);
void lc_store_destroy(lc_store* store);

/* Forgets every version (a log store reuses its arena from the start).
 * Errors: STATE (a pending version is still being copied). */
lc_status lc_store_clear(lc_store* store);

int64_t lc_store_num_versions(const lc_store* store);

/* A store's arena and its use. */
typedef struct {
    const void* arena;         /* pinned host base address of the arena         */
    uint64_t capacity;         /* arena bytes                                   */
    uint64_t excluded_bytes;   /* bytes kept out of use (lc_store_exclude)      */
    uint64_t used_bytes;       /* bytes held by versions, pending or durable    */
    int32_t versions_per_layer;
    int32_t reserved;
    uint64_t avoided_bytes;    /* slow bytes left in use by lc_store_check_dma  */
} lc_store_info;

/* Errors: INVALID_ARG (NULL). */
lc_status lc_store_get_info(const lc_store* store, lc_store_info* out);
lc_status lc_store_get_version(const lc_store* store, int64_t index, lc_version* out);

/* Takes bytes [offset, offset + bytes) of the store's arena (widened to
 * whole 4096-byte granules) out of use: no later version is placed there.
 * Log and newest-only stores; the range must hold no version.  Excluded
 * ranges stay excluded across lc_store_clear.  A log store places each layer
 * block at the next offset whose block touches no excluded range.
 * Errors: INVALID_ARG (ring store, range outside the arena), STATE (a
 * version lies in the range). */
lc_status lc_store_exclude(lc_store* store, uint64_t offset, uint64_t bytes);

/* Pinned host memory is not uniform for the GPU: on a shared host some of
 * its pages can take device copies at a small fraction of the link rate,
 * and not all the time (measured here: a fixed set of a few GB of an 80 GB
 * pinned arena copying at 15-60 GB/s in about half of the passes over it,
 * the rest at 193 GB/s in every pass).  This times `passes` device->host
 * copies into every region_bytes region of an empty log or newest-only
 * store (from a device buffer on ctx's device).  A region is slow if its
 * slowest pass ran below min_fraction times the median of the regions'
 * fastest passes.  The slow regions are excluded (lc_store_exclude) one at
 * a time, slowest first (the lower index first on a tie), except that one
 * whose exclusion would leave no room for a step that persists every layer
 * stays in use: every layer's block in layer order from offset 0 (log
 * store), or each block size's slots for its layers plus the spare
 * (newest-only store).  A store that lacks that room before the call loses
 * every slow region.  The slow regions left in use are avoided: a log store
 * places a step's blocks off them whenever the whole step fits that way,
 * and a newest-only store lays its slots out off them whenever its layers'
 * slots and spares fit that way (lc_store_info.avoided_bytes); each call
 * replaces the previous call's avoided regions.  region_bytes: 0 (256 MiB)
 * or a multiple of 4096 in [1 MiB, 1 GiB]; passes: 0 (4) or 1..64.
 * rates_out (host, nullable): each of the ceil(capacity / region_bytes)
 * regions' slowest GB/s; excluded_out (nullable): bytes excluded.
 * Overwrites the arena; blocks (bounded by ctx's timeout_ms).
 * Errors: INVALID_ARG, STATE (the store holds versions), TIMEOUT, CUDA,
 * OOM. */
lc_status lc_store_check_dma(lc_store* store, lc_ctx* ctx, uint64_t region_bytes, int32_t passes,
                             double min_fraction, double* rates_out, int64_t rates_cap, uint64_t* excluded_out);

/* §3.5 reconstruction plan: pick_out[l] = index of the durable version of
 * layer l with the largest step <= t_fail (the newer record on a tie), or
 * -1.  Returns NOT_FOUND if some layer has none. */
lc_status lc_store_plan(const lc_store* store, int64_t t_fail, int64_t* pick_out);

/* --- file tier of the store: §3.5 metadata-driven recovery -------------- *
 * A checkpoint directory holds two append-only files.
 *   blocks.lcb   : packed layer blocks (the §3.1 layout of lc_pack_*), each
 *                  starting on a 4096-byte boundary.
 *   manifest.lcm : a 64-byte header, then one 64-byte record per block.
 * All integers are little-endian.  Header: "LCMH", format 1 (u32), nlayers
 * (i32), layout CRC (u32: CRC-32C of the nlayers block sizes as u64), zeros,
 * and at byte 60 the CRC-32C of bytes [0, 60).  Record: "LCVR", layer (i32),
 * step (i64), offset in blocks.lcb (u64), bytes (u64), CRC-32C of the block
 * (u32), layout CRC (u32), zeros, and at byte 60 the CRC-32C of [0, 60).
 * A block is written (and synced, if asked) before its record, so a record
 * never names a block that is not there; the log ends at the first short or
 * invalid record (a torn append), which the next append overwrites.  The
 * recovery reads the records only -- the metadata -- to choose, per layer,
 * the newest version at or before the failure step (§3.5), and then reads
 * just those blocks, checking each against its CRC. */

/* CRC-32C (Castagnoli, reflected polynomial 0x82F63B78, initial value and
 * final XOR 0xFFFFFFFF) of data[0, nbytes), continuing from `crc` (0 to
 * start; crc32c(B, crc32c(A, 0)) is the CRC of A followed by B).  Host
 * memory; large inputs are split over the host's cores. */
uint32_t lc_crc32c(const void* data, uint64_t nbytes, uint32_t crc);

/* Appends to directory `dir` (created if missing) every durable version of
 * `store` whose (layer, step) the manifest does not hold yet, in version
 * order.  sync != 0: each block and each record is fdatasync'd before the
 * next write.  bytes_written (nullable): block bytes appended.  Call it from
 * the thread that drives the store's context, between steps.
 * Errors: INVALID_ARG (dir holds another layout, or is unusable), STATE
 * (the manifest's header is corrupt). */
lc_status lc_store_persist_dir(lc_store* store, const char* dir, int32_t sync, uint64_t* bytes_written);

/* §3.5 / Eq. 8 from a checkpoint directory: for every layer of ctx's layout
 * the version with the largest step <= t_fail (the later record on a tie)
 * whose record and block CRCs check out; a version whose block fails its CRC
 * is passed over for the next older one.  Reads only those blocks, into a
 * new log store (*out, one durable version per layer, owned by the caller:
 * lc_store_destroy) that lc_restore(ctx, *out, t_fail, ...) then scatters
 * onto the device.  layer_steps_out: host, nlayers (nullable).
 * Errors: NOT_FOUND (a layer has no intact version <= t_fail), INVALID_ARG
 * (another layout, no manifest), STATE, OOM. */
lc_status lc_store_load_dir(lc_ctx* ctx, const char* dir, int64_t t_fail, lc_store** out,
                            int64_t* layer_steps_out);

/* One manifest record as read back. */
typedef struct {
    int32_t layer;
    int32_t intact;          /* block CRC checked and equal (verify_blocks), else 1 */
    int64_t step;
    uint64_t offset;         /* in blocks.lcb */
    uint64_t bytes;
    uint32_t block_crc;
    uint32_t layout_crc;
} lc_manifest_record;

/* Reads the manifest of `dir` without a GPU.  out (nullable) receives up to
 * cap valid records in file order; *n_out = the number of valid records;
 * *nlayers_out and *layout_crc_out from the header; *torn_out = 1 if the log
 * ends in a short or invalid record.  verify_blocks != 0 reads every block
 * and sets `intact` from its CRC.  Any out pointer may be NULL.
 * Errors: INVALID_ARG (no manifest), STATE (corrupt header). */
lc_status lc_manifest_read(const char* dir, int32_t verify_blocks, lc_manifest_record* out, int64_t cap,
                           int64_t* n_out, int32_t* nlayers_out, uint32_t* layout_crc_out, int32_t* torn_out);

/* --- the measure without any device allocation -------------------------- */

/* Limits of lc_measure_noalloc (its scratch is a fixed-size array). */
#define LC_NOALLOC_MAX_SEGMENTS 512
#define LC_NOALLOC_MAX_LAYERS 512
#define LC_NOALLOC_SCRATCH_BYTES (192u * 1024u)

/* The paper has no counterpart to this entry point; it exists for callers
 * that cannot allocate device memory.  Some host programs must not call
 * cudaMalloc once they are running: a framework that owns every byte of
 * the GPU through its own memory pool, a process whose device footprint is
 * fixed at start-up, or code where an allocation could synchronize the
 * device at a bad moment.  Such a caller can still get the per-layer sums
 * that lc_measure computes from this call, without an lc_ctx.
 *
 * Computes, on `cuda_stream` of `device`, the same per-layer sums as
 * lc_measure: sums_out[3*l] = sum |W - R|, sums_out[3*l+1] = sum |R|,
 * sums_out[3*l+2] = element count of layer l, for the segments `segs` (host
 * array of nseg lc_segment in any layer order, the layout rules of
 * lc_register_layout: snap is required and must not alias w; it is only
 * read, exp_avg / exp_avg_sq are ignored).  A layer's segments are summed in
 * their order within `segs`.  sums_out: caller-owned device memory of
 * 3*nlayers fp64, 8-byte aligned.  Asynchronous.  The segment table and the
 * work partition travel to the device inside the call's own kernel
 * launches, so the host array may be reused, and nothing on the host is
 * read, once the call has returned.
 *
 * Memory: the call allocates nothing.  Its scratch (tables, partial sums,
 * completion counter) lives in one static device array of
 * LC_NOALLOC_SCRATCH_BYTES that every GPU which loads the library holds
 * until the process exits.  The first call on a device looks up that
 * array's device address (cudaGetSymbolAddress) with the device current;
 * make that first call before any stream capture.  All calls share the
 * array: calls that overlap on the GPU (different streams, or different
 * host threads, without ordering between them) race and give wrong sums.
 *
 * Errors: INVALID_ARG (layout, pointers), CAPACITY (nseg above
 * LC_NOALLOC_MAX_SEGMENTS or nlayers above LC_NOALLOC_MAX_LAYERS), CUDA. */
lc_status lc_measure_noalloc(int device, void* cuda_stream, const lc_segment* segs,
                             int32_t nseg, int32_t nlayers, double* sums_out);

#ifdef __cplusplus
}
#endif
#endif /* LAYERCHECK_H */
