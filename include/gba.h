/*
 * gba.h - C ABI of libgba: the GBA aggregate-and-apply step on one GB300 GPU.
 *
 * GBA (Global Batch gradients Aggregation, arXiv 2205.11048) keeps the global
 * batch of synchronous training while workers push asynchronously: the
 * parameter server buffers (gradient, token) messages until the buffered local
 * batches reach the global batch, excludes gradients whose token staleness
 * exceeds a threshold (Sec. 4.1, Eq. (1)), and applies the aggregate once per
 * global step (Alg. 2, push responding threads).
 *
 * Conventions for every entry point:
 *  - No exception crosses this ABI.  Functions return a gba_status (or a
 *    documented integer); GBA_OK is 0, errors are negative.
 *  - A handle is used by one host thread at a time.
 *  - All GPU work of a handle is issued on the stream given to gba_create, in
 *    submission order; results are visible to work ordered after it on that
 *    stream, or after gba_sync.
 *  - Device errors found by a kernel (an id out of range, a bounded wait that
 *    gave up) are latched: the next gba_try_apply or gba_sync returns the code
 *    and the handle refuses further steps with GBA_E_STATE.
 */
#ifndef GBA_H_
#define GBA_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct gba_handle gba_handle; /* opaque, owned by the library */

typedef enum {
  GBA_OK = 0,
  GBA_E_ARG = -1,            /* invalid argument; nothing was changed */
  GBA_E_ID_RANGE = -2,       /* a DIRECT id was outside [0, rows): the step was not applied */
  GBA_E_OOM = -3,            /* device or pinned host allocation failed */
  GBA_E_CUDA = -4,           /* a CUDA runtime call failed (see gba_last_error) */
  GBA_E_DEVICE_TIMEOUT = -5, /* a bounded device-side wait gave up */
  GBA_E_STATE = -6,          /* the handle failed earlier and accepts no more steps */
  GBA_E_FULL = -7            /* the gradient buffer is full; apply, then push again */
} gba_status;

typedef enum { GBA_ADAGRAD = 0, GBA_ADAM = 1 } gba_optimizer;

/* id -> row mapping of a table:
 * DIRECT: the id is the row and must satisfy 0 <= id < rows;
 * MODULO: row = (uint64_t)id % rows (hashing trick; colliding ids share a row);
 * HASH:   an expandable hash table of 64-bit ids (the paper's models run on
 *         DeepRec's expandable hash tables, Sec. 5.1): every distinct id gets a
 *         row of its own, created when the id is first pushed and initialised
 *         from the id (element id * dim + j of the table's counter-based
 *         stream), so an id's values do not depend on where it is stored.
 *         `rows` is the initial capacity (rounded up to a power of two, at
 *         least 1024, at most 2^30); the table doubles before a step that
 *         could fill more than half of it.  The id INT64_MIN is reserved
 *         (a step containing it fails with GBA_E_ID_RANGE).  The arrays of
 *         gba_get_table are indexed by slot: use gba_table_capacity for their
 *         size and gba_lookup_rows for the slot of an id; growth moves rows
 *         and replaces the arrays, so take the pointers again after a step. */
typedef enum { GBA_ID_DIRECT = 0, GBA_ID_MODULO = 1, GBA_ID_HASH = 2 } gba_id_mode;

/* Optimizer of a table or of the dense parameters.  Table 1 of the paper names
 * Adagrad and Adam; the update rules are the textbook ones, one IEEE float
 * operation at a time:
 *   Adagrad: a += g*g;  w -= (lr*g) / sqrt(a)            (a starts at adagrad_init_acc > 0)
 *   Adam:    m = b1*m + (1-b1)*g;  v = b2*v + (1-b2)*(g*g);
 *            w -= (lr*(m/bc1)) / (sqrt(v/bc2) + eps),  bc_i = 1 - b_i^t, t = global step + 1 */
typedef struct {
  int32_t kind;            /* gba_optimizer */
  float lr;
  float adagrad_init_acc;  /* Adagrad only; paper default 0.1 */
  float beta1, beta2, eps; /* Adam only; 0.9, 0.999, 1e-8 */
} gba_opt_desc;

/* One embedding table: rows x dim float32 weights plus optimizer state and a
 * per-row step tag (Alg. 2: each ID carries the global step at which it was last
 * updated). */
typedef struct {
  int64_t rows;            /* >= 1; the sum of rows over all tables must be < 2^32 */
  int32_t dim;             /* 1 .. 256 */
  int32_t id_mode;         /* gba_id_mode */
  int64_t max_ids_per_msg; /* upper bound on one message's ids for this table (sizes the buffers) */
  gba_opt_desc opt;
} gba_table_desc;

/* Staleness rule (Sec. 4.1 Eq. (1)): a gradient with staleness s is kept iff
 * s <= iota; staleness = max(0, reference - token).
 *   row_staleness 0: rows use the row's step tag as the reference (Alg. 2),
 *                 1: rows use the current step k, like the dense gradient.
 *   sparse_denominator 0: divide a row's kept sum by the number of messages in
 *                 the global batch that contain the row (Alg. 2: the workers
 *                 whose batches held the ID), 1: by the kept ones, 2: by M.
 *   decay 0: a kept gradient weighs 1 (Eq. (1) as printed);
 *         1: a kept gradient of staleness s weighs lambda^s (Sec. 4.1 allows
 *            other decay strategies; lambda^s is s products in double, rounded
 *            to float once); needs 0 < lambda <= 1 and iota <= 1023.
 *   drop_latest: Hop-BW's backup workers (Sec. 5.1): the last drop_latest
 *            popped messages of every step weigh 0 (dense and rows); 0: none.
 * iota = INT32_MAX keeps every gradient (BSP). */
typedef struct {
  int32_t iota;
  int32_t row_staleness;
  int32_t sparse_denominator;
  int32_t decay;
  float lambda;
  int32_t drop_latest;
} gba_staleness_desc;

/* The sparse part of one message for one table: n ids and n x dim gradient rows
 * (row-major float32). */
typedef struct {
  const int64_t* ids;
  int64_t n;
  const float* rows;
} gba_sparse_grad;

/* Counters accumulated over all applied steps (Table 3 reports the number of
 * excluded batches and the average / max staleness). */
typedef struct {
  int64_t steps;
  int64_t msgs_kept, msgs_dropped;          /* dense decisions */
  int64_t dense_stale_sum, dense_stale_max; /* over all popped messages */
  int64_t pairs, pairs_dropped;             /* distinct (message, row) pairs */
  int64_t row_stale_sum, row_stale_max;     /* over those pairs */
  int64_t occurrences;                      /* id occurrences */
  int64_t rows_touched, rows_applied;       /* unique rows; those that took a step */
  int64_t occurrences_kept;                 /* occurrences whose gradient was aggregated */
} gba_stats_t;

/* Per kernel class: launches and device time summed since timing was enabled. */
/* indices into gba_kernel_times_t: K1 message weights; K2 sort (digit
 * histograms, one onesweep pass per key digit); K3 segment scan (decisions,
 * row records, kept list); K3+K4 long rows (chunked sums and their update);
 * K3+K4 row sums and update; K5 dense update; table init. */
enum {
  GBA_K_WEIGHTS = 0, GBA_K_SORT_HIST = 1, GBA_K_SORT_PASS = 2, GBA_K_SEG_SCAN = 3,
  GBA_K_ROW_LONG = 4, GBA_K_ROW_APPLY = 5, GBA_K_DENSE = 6, GBA_K_INIT = 7,
  GBA_K_OTHER = 8, GBA_K_COUNT = 9
};
typedef struct {
  int64_t launches[GBA_K_COUNT];
  double ms[GBA_K_COUNT];
} gba_kernel_times_t;

/*
 * gba_create - allocate the parameter-server state on the current device.
 *
 * tables[n_tables]   table descriptions (n_tables may be 0).
 * dense_size         number of dense float32 parameters (may be 0).
 * dense_opt          optimizer of the dense parameters (may be NULL if dense_size is 0).
 * global_batch       G: a step is applied once the buffered local batches sum to >= G
 *                    (Sec. 4.1: G_a = B_a * M equals the synchronous B_s * N_s).
 * max_buffered_msgs  capacity of the gradient buffer, in messages (>= 1).
 * st                 staleness rule (NULL: iota = INT32_MAX, tags, encountered,
 *                    weight 1, nothing ignored).
 * init_seed          weights are initialised from a counter-based hash of
 *                    (seed, table, element); optimizer state from the descriptors.
 * cuda_stream        cudaStream_t for all work of the handle; NULL makes a new one.
 * out                receives the handle.
 * Returns GBA_E_ARG for invalid descriptions, GBA_E_OOM / GBA_E_CUDA on failure.
 */
gba_status gba_create(const gba_table_desc* tables, int32_t n_tables, int64_t dense_size,
                      const gba_opt_desc* dense_opt, int64_t global_batch,
                      int32_t max_buffered_msgs, const gba_staleness_desc* st,
                      uint64_t init_seed, void* cuda_stream, gba_handle** out);

/*
 * gba_push - store one worker message in the gradient buffer (Alg. 2: "store
 * the gradients with the token to the gradient buffer").
 *
 * token        the global step the worker's batch was issued at (>= 0; a
 *              token ahead of the current step counts as staleness 0).
 * per_table    n_tables entries; ids/rows may be device or host pointers
 *              (host memory should be pinned for the copy to be asynchronous).
 * dense_grad   dense_size floats, device or host.
 * local_batch  the message's local batch size B (>= 1).
 * The data are copied on the handle's stream; the caller may reuse its buffers
 * once that copy is complete (stream order).  GBA_E_FULL when the buffer holds
 * max_buffered_msgs messages; GBA_E_ARG for n > max_ids_per_msg or NULL data.
 */
gba_status gba_push(gba_handle* h, int64_t token, const gba_sparse_grad* per_table,
                    const float* dense_grad, int32_t local_batch);

/*
 * gba_push_ref - like gba_push, but the library only records the pointers:
 * the device buffers must stay valid and unmodified until the step that pops
 * the message has completed on the stream.  Pointers must be device memory;
 * dense_grad must be 16-byte aligned, and rows too when dim is a multiple of 4.
 */
gba_status gba_push_ref(gba_handle* h, int64_t token, const gba_sparse_grad* per_table,
                        const float* dense_grad, int32_t local_batch);

/*
 * gba_try_apply - if the buffered local batches reach the global batch, pop the
 * oldest messages that do (Alg. 2 takes N_a gradients off the buffer), enqueue
 * one global step on the stream and return 1; otherwise return 0.  The step:
 *   Eq. (1) weights per message; rows deduplicated by id (radix sort);
 *   per row: decay by the row's tag vs the token, sum of kept gradients divided
 *   by the denominator, optimizer, tag := k + 1 (rows with no kept gradient are
 *   left untouched); dense: sum of kept gradients / M, optimizer (always).
 * A negative return is a gba_status (a latched device error surfaces here).
 */
int32_t gba_try_apply(gba_handle* h);

/* gba_pull_version - the number of global steps applied so far (k).  Sec. 4.1
 * defines a batch's token as the global step at which it is handed to a
 * worker, and Alg. 2 (pull responding) hands the token out with the
 * parameters; a worker that takes its token from here is counted as stale by
 * k' - k when its gradient is applied at step k'.  NULL handle: -1. */
int64_t gba_pull_version(gba_handle* h);

/* gba_sync - wait for all work of the handle, then report any latched device error. */
gba_status gba_sync(gba_handle* h);

/* gba_get_table / gba_get_dense - device pointers to the state (borrowed, valid
 * until gba_destroy): weights [rows*dim], slot0 (Adagrad accumulator or Adam m),
 * slot1 (Adam v, NULL for Adagrad), per-row step tags [rows]. */
gba_status gba_get_table(gba_handle* h, int32_t t, float** w, float** slot0, float** slot1,
                         int32_t** ver);
gba_status gba_get_dense(gba_handle* h, float** w, float** slot0, float** slot1);

/* gba_stats - synchronise and copy the accumulated counters. */
gba_status gba_stats(gba_handle* h, gba_stats_t* out);

/* gba_last_error - text of the last failure of this handle ("" if none). */
const char* gba_last_error(gba_handle* h);

/* gba_destroy - wait for outstanding work and free everything (NULL is a no-op). */
void gba_destroy(gba_handle* h);

/*
 * gba_set_overlap - when on, gba_try_apply does not order the handle's stream
 * after the step it enqueues, so the next step's message weights and sort can
 * run while this step's segment-sum and dense update finish (steps still apply
 * in order: each step's row update follows the previous one's).  The caller
 * then sees a step's results after gba_sync (or any call that synchronises).
 * Copying pushes still wait for every earlier step.  Default off: every step is
 * complete, in the handle's stream order, before later work on that stream.
 */
gba_status gba_set_overlap(gba_handle* h, int32_t on);

/*
 * gba_pull - pull responding (Alg. 2: "look up the embedding tables based on
 * the IDs for the embedding parameters" and send them to the worker).
 *
 * t      table index.
 * ids    n device int64 ids (8-byte aligned), mapped to rows as in the table's
 *        id_mode.
 * out    n x dim device float32 (row-major), receives the rows' current
 *        weights as of every step enqueued before this call.
 * Enqueued on the handle's stream (after joining any overlapping steps); the
 * rows are in out for work ordered after it on that stream.  A DIRECT id
 * outside [0, rows) gets a row of zeros and is latched like a step's id error
 * (the next gba_sync / gba_try_apply returns GBA_E_ID_RANGE).  GBA_E_ARG for a
 * bad table index or NULL pointers with n > 0.
 */
gba_status gba_pull(gba_handle* h, int32_t t, const int64_t* ids, int64_t n, float* out);

/*
 * The token list (Sec. 4.1; Alg. 2 token generation and pull responding
 * threads): a queue of tokens handed to workers with their batches.  Token
 * values start at 0 and each repeats `repeats` (M) times, so the i-th token
 * fetched is floor(i / M).  Whenever the queue holds fewer tokens than
 * `workers`, new tokens are appended until it holds `workers` (the paper's
 * refill, done under a lock).  gba_fetch_token may be called from any number
 * of host threads at once.  The list needs no GPU.
 *
 * gba_token_list_create   GBA_E_ARG if repeats < 1 or workers < 1.
 * gba_fetch_token         takes the head of the queue into *token.
 * gba_token_list_state    tokens queued now, and fetched so far.
 */
typedef struct gba_token_list gba_token_list;
gba_status gba_token_list_create(int64_t repeats, int32_t workers, gba_token_list** out);
gba_status gba_fetch_token(gba_token_list* tl, int64_t* token);
gba_status gba_token_list_state(gba_token_list* tl, int64_t* queued, int64_t* fetched);
void gba_token_list_destroy(gba_token_list* tl);

/* gba_table_capacity - the rows the arrays of table t hold now (for a HASH
 * table, its current number of slots). */
gba_status gba_table_capacity(gba_handle* h, int32_t t, int64_t* rows);

/* gba_lookup_rows - for a HASH table, the row (slot) of each of n device
 * int64 ids into n device int64 (-1 for an id not in the table), on the
 * handle's stream after every step enqueued so far.  GBA_E_ARG for other
 * tables. */
gba_status gba_lookup_rows(gba_handle* h, int32_t t, const int64_t* ids, int64_t n,
                           int64_t* rows_out);

/*
 * gba_set_eager_dense - when on, a pushed message's dense gradient is added to
 * the compensated sum of the global step it belongs to at push time, instead
 * of being kept until that step (the memory saving that the discussion of
 * Alg. 2 points out: the tokens fix the weights, so part of the weighted sum
 * may be formed before the step).  The FIFO fixes each message's step (the
 * shortest prefix of buffered local batches reaching G), so its weight
 * (Eq. (1) or the decay strategy) is known when it arrives.  Sums are formed
 * in arrival order, the order of the buffered mode, so results are identical.
 * The dense part of the gradient buffer shrinks from one gradient per
 * buffered message to one accumulator pair per pending global step (at most 8
 * pending steps: a push that would need a ninth returns GBA_E_FULL).  Row
 * gradients stay buffered (their decay needs the per-ID tags as of their
 * step).  Only while no message is buffered (else GBA_E_STATE); GBA_E_ARG with
 * drop_latest > 0, since the latest messages of a step are unknown at push.
 * Pushes then launch a kernel on the handle's stream; push_ref's dense buffer
 * may be reused once that kernel has run.
 */
gba_status gba_set_eager_dense(gba_handle* h, int32_t on);

/*
 * gba_join - order the handle's stream after every step enqueued so far (their
 * segment-sum, row update and dense update included), without waiting on the
 * host.  Work the caller enqueues on that stream afterwards, an event recorded
 * there for instance, sees the results of every applied step.  Needed only
 * with overlap on; with overlap off each gba_try_apply already does this.
 */
gba_status gba_join(gba_handle* h);

/* ---- instrumentation and test entry points ----------------------------- */

/* gba_set_timing - when on, every kernel launch is bracketed by CUDA events on
 * its stream; gba_kernel_times synchronises and returns the sums. */
gba_status gba_set_timing(gba_handle* h, int32_t on);
gba_status gba_kernel_times(gba_handle* h, gba_kernel_times_t* out);

/* gba_set_debug - when on, each step also records the dedup result so that
 * gba_debug_segments can return it (costs one extra write per unique row). */
gba_status gba_set_debug(gba_handle* h, int32_t on);

/*
 * gba_debug_segments - dedup output of the last applied step (debug must have
 * been on for it).  Host buffers of capacity cap receive, per unique row in
 * increasing (table, row) order: table[i], row[i], count[i] (messages that
 * contain the row) and kept[i] (kept occurrences).  *n_unique receives the
 * number of unique rows (GBA_E_ARG if it exceeds cap).
 */
gba_status gba_debug_segments(gba_handle* h, int64_t cap, int32_t* table, int64_t* row,
                              int64_t* count, int64_t* kept, int64_t* n_unique);

/* gba_debug_sorted - the last step's sorted keys (global row = sum of the rows
 * of earlier tables + row) and occurrence indices, into host buffers of
 * capacity cap; *n receives the number of occurrences. */
gba_status gba_debug_sorted(gba_handle* h, int64_t cap, uint32_t* keys, uint32_t* occ,
                            int64_t* n);

/* gba_debug_keep - message weights f (Eq. (1)) of the last step, in pop order. */
gba_status gba_debug_keep(gba_handle* h, int32_t cap, int32_t* keep, int32_t* M);

/* gba_debug_set_wait_limit - the time (ns) after which a device-side wait of
 * this handle gives up and latches GBA_E_DEVICE_TIMEOUT (default 2e9). */
gba_status gba_debug_set_wait_limit(gba_handle* h, int64_t ns);

/* gba_debug_withhold_dense_copies - test hook for the bounded waits of K5 in
 * the buffered dense mode: with on = 1 the dense kernel's producer issues no
 * copies, so every consumer wait runs out after the handle's wait limit and
 * the step reports GBA_E_DEVICE_TIMEOUT (from gba_try_apply or gba_sync); the
 * dense parameters are then undefined and the handle is failed, as after any
 * device timeout.  on = 0 restores normal operation.  GBA_E_ARG for other
 * values. */
gba_status gba_debug_withhold_dense_copies(gba_handle* h, int32_t on);

/*
 * gba_selftest_wait_timeout - run the library's bounded device wait on a flag
 * that nothing sets, with the given limit, on the given stream (NULL = default
 * stream), and return the status the kernel reports: GBA_E_DEVICE_TIMEOUT when
 * the wait gave up as designed.
 */
gba_status gba_selftest_wait_timeout(int64_t limit_ns, void* cuda_stream);

/*
 * gba_sort_ids_static - sort one batch of ids by row without allocating.
 *
 * The paper has no counterpart to this entry point.  It serves callers that
 * must not allocate device memory at the moment they sort: a runtime that
 * reserved all device memory up front and hands out no more, or an allocator's
 * own hook, which cannot call back into cudaMalloc.  It runs the same
 * histogram and onesweep radix-sort kernels as gba_try_apply, but takes its
 * scratch from one fixed device array of GBA_STATIC_SORT_BYTES bytes that is
 * part of the library image: every GPU that loads the library holds that array
 * until the process exits.  The call itself allocates nothing (no cudaMalloc,
 * cudaFree or allocating library routine).
 *
 * ids        n device int64 ids; row = id (id_mode DIRECT, 0 <= id < rows) or
 *            (uint64)id % rows (MODULO).
 * n          0 .. GBA_STATIC_SORT_MAX_IDS; larger n returns GBA_E_ARG.
 * rows       1 .. 2^32 - 2.
 * rows_out   n device uint32: the rows of the ids in ascending order.
 * order_out  n device uint32: order_out[i] is the input index of rows_out[i];
 *            equal rows keep their input order (stable).
 * cuda_stream  the stream to run on (NULL: the legacy default stream).
 *
 * The call is synchronous: it enqueues its kernels on the stream, waits for the
 * stream to finish, and returns GBA_OK, GBA_E_ID_RANGE (a DIRECT id outside
 * [0, rows)), GBA_E_DEVICE_TIMEOUT (a bounded wait of the sort gave up) or
 * GBA_E_CUDA (a CUDA call failed, or a CUDA error was already pending on the
 * calling thread; a pending error is left in place for its owner).  rows_out and order_out
 * hold the sorted result only when GBA_OK is returned; after an error their
 * contents are undefined.
 * The first call on a device, with that device current, looks up the array's
 * device address.  All calls share the one array, which keeps the previous
 * call's contents (the counters that must start at zero are cleared at the
 * start of each call): calls whose work overlaps on the GPU (two streams, or
 * two host threads) race and give wrong results.
 */
#define GBA_STATIC_SORT_MAX_IDS (1 << 20)
#define GBA_STATIC_SORT_BYTES 9441392
gba_status gba_sort_ids_static(const int64_t* ids, int64_t n, int64_t rows, int32_t id_mode,
                               uint32_t* rows_out, uint32_t* order_out, void* cuda_stream);

/* gba_device_binary_version - the compute capability of the device code the
 * library's kernels run from on the current device, as major * 10 + minor
 * (103 for sm_103a), or GBA_E_CUDA when no device code could be loaded. */
int32_t gba_device_binary_version(void);

/* gba_version_string - library build identification. */
const char* gba_version_string(void);

#ifdef __cplusplus
}
#endif

#endif /* GBA_H_ */
