/*
 * mlkv_gpu.h -- C ABI of the GB300 batched embedding key-value store.
 *
 * One table = an open-addressing hash index (64-bit key -> dense row id) plus
 * fp32 rows and fp32 Adagrad state, all resident in HBM.  The calls follow the
 * storage interface of MLKV (arXiv 2504.01506):
 *   Section 3.1  Open(model_id, dim, staleness_bound), Get(keys) -> values,
 *                Put(keys, values) (upsert), Lookahead(keys, dest);
 *   Section 3.2  step 8 and Figure 2: the gradient update is a per-key
 *                read-modify-write of the stored vectors (Put or Rmw of
 *                values + emb_optimizer(gradients)).
 * The optimizer is element-wise Adagrad, one step per distinct key on the sum
 * of that key's gradients in the batch (the gradient of the embedding map E of
 * Section 2.1):
 *       G[r] += g*g ;  w[r] -= lr * g / (sqrt(G[r]) + eps)
 *
 * Conventions shared by every call
 *   - Pointers named d_* are DEVICE pointers owned by the caller; pointers
 *     named h_* are HOST pointers owned by the caller (pinned memory makes
 *     the copies asynchronous; pageable memory works but the copy blocks).
 *     Buffers must stay valid until the stream has executed the call.
 *   - Keys are int64 reinterpreted as uint64.  The key -1 (all bits set) is
 *     reserved for empty index slots: a kernel that meets it records
 *     MLKV_ERR_INVALID and treats that lookup as absent (NaN output, no
 *     update, never inserted).
 *   - Row-major layouts: values, gradients and outputs are [n][dim] fp32.
 *   - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *     default stream).  All calls of one table share its scratch memory, so
 *     issue them on one stream, or order them with events.  A table may be
 *     used from one host thread at a time.
 *   - Errors a host check finds are returned at once and nothing is enqueued.
 *     Errors a kernel finds (MLKV_ERR_FULL, MLKV_ERR_PROBE_LIMIT,
 *     MLKV_ERR_NOT_FOUND, MLKV_ERR_INVALID for the reserved key) are sticky:
 *     they are recorded in the table's status word, returned by mlkv_sync and
 *     by later calls once the GPU has reached the failing call, and cleared by
 *     mlkv_clear_status.
 *   - n == 0 is a no-op that returns MLKV_OK (after the argument checks).
 *   - No call allocates device memory except mlkv_open (the table, its index,
 *     its scratch sized for max_batch) and the first *_host call (staging
 *     sized for max_batch).  Every loop inside a kernel is bounded (the probe
 *     limit, the tier's sweep limit).  The only waits are the grid barriers of
 *     the kernel that gives new keys their rows, between the blocks of that
 *     one grid (one block per SM; the next kernel may launch only after them),
 *     bounded: one that runs out records MLKV_ERR_TIMEOUT.
 *   - Each call that enqueues work, and mlkv_open / close / sync /
 *     clear_status, is an NVTX range named after the call ("mlkv_get",
 *     "mlkv_apply_grad", ...), for timeline tools; the kernels it launches
 *     fall inside it.
 */
#ifndef MLKV_GPU_H
#define MLKV_GPU_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes. */
#define MLKV_OK 0
#define MLKV_ERR_INVALID 1     /* bad argument: null pointer, n < 0, n > max_batch, reserved key */
#define MLKV_ERR_UNSUPPORTED 2 /* a configuration this build does not provide */
#define MLKV_ERR_CUDA 3        /* a CUDA runtime call failed; mlkv_last_error has the text */
#define MLKV_ERR_NOMEM 4       /* device or pinned allocation failed */
#define MLKV_ERR_FULL 5        /* more distinct keys than `capacity` */
#define MLKV_ERR_PROBE_LIMIT 6 /* an index probe exceeded the probe bound */
#define MLKV_ERR_NOT_FOUND 7   /* absent key and insert_on_miss == 0 */
#define MLKV_ERR_TIMEOUT 8     /* a bounded wait inside a kernel ran out: the grid barriers of the
                                  miss path (new keys) of a call, between blocks of one grid */

/* Largest dimension the row kernels take (8 vectors per lane of a warp). */
#define MLKV_MAX_DIM 1024  /* dim > 256 needs dim % 4 == 0 */

/* Segments (runs of one key in a gradient batch) of at most this many
 * occurrences are summed by one lane group in occurrence order, so their
 * Adagrad step is the same op sequence as a sequential fp32 statement of it.
 * Longer segments are summed in chunks (64 lookups in calls of at least 2^19
 * lookups, 16 in smaller ones) with compensated (TwoSum) additions and the
 * chunks' (sum, compensation) pairs combined in a fixed order, the sum rounded
 * once: deterministic run to run and within about one rounding of the exact
 * sum, not the sequential fp32 rounding. */
#define MLKV_SEQ_SEGMENT_MAX 32

/* Flags of mlkv_config.flags. */
#define MLKV_IDENTITY_HASH 2u  /* index slot = key mod 2^k (tests of long probe chains only) */

/* Longest probe sequence of the index; a longer one records MLKV_ERR_PROBE_LIMIT. */
#define MLKV_PROBE_LIMIT 1024

/* staleness_bound values (MLKV Section 3.3.1): 0 is bulk-synchronous, this one
 * asynchronous (no bound), any other stale-synchronous.  A bound above
 * MLKV_MAX_STALENESS is kept as MLKV_MAX_STALENESS: a tighter bound, which
 * meets the one asked for. */
#define MLKV_STALENESS_ASYNC INT64_MAX
#define MLKV_MAX_STALENESS 64

/*
 * Open of MLKV Section 3.1: Open(model_id, dim, staleness_bound).  model_id
 * maps to the returned handle; one handle per table.
 */
typedef struct mlkv_config {
    int32_t dim;             /* embedding dimension d, 1..MLKV_MAX_DIM */
    int32_t insert_on_miss;  /* 1: Get / apply_grad of an absent key insert it with the init row */
    int64_t capacity;        /* maximum number of distinct keys (rows), >= 1, < 2^31 */
    int64_t max_batch;       /* maximum n of one call, >= 1, < 2^30 */
    float lr;                /* Adagrad learning rate */
    float eps;               /* Adagrad epsilon, added to sqrt(G) */
    float state_init;        /* Adagrad state of a new row */
    float init_lo, init_hi;  /* a new row is drawn U[init_lo, init_hi) by the counter-based init */
    uint64_t seed;           /* seed of the counter-based init */
    int64_t staleness_bound; /* MLKV's consistency bound s (Section 3.3.1), >= 0: 0 bulk-
                                synchronous; MLKV_STALENESS_ASYNC asynchronous; any other
                                stale-synchronous (HBM-resident tables; see below) */
    int64_t hbm_cache_rows;  /* 0: rows + state resident in HBM.  > 0: rows + state live in host
                                memory (the tier) and this many rows are cached in HBM; it must be
                                >= 2 * max_batch + 64 (a call and a look-ahead in flight) */
    uint32_t flags;          /* 0 or MLKV_IDENTITY_HASH */
    uint32_t reserved;       /* 0 */
} mlkv_config;

typedef struct mlkv_table mlkv_table; /* opaque; owned by the library */

/* Row initialisation of a new key k, element j (any implementation reproduces it):
 *   x = splitmix64(seed ^ splitmix64(k ^ (j * 0x9E3779B97F4A7C15)))
 *   v = init_lo + ((x >> 40) * 2^-24) * (init_hi - init_lo)   (fp32, each op rounded)
 * where splitmix64(z) is the output of a SplitMix64 generator (Steele, Lea &
 * Flood 2014) whose state is z.  State starts at state_init. */

/* Streams and graphs.  Every call that takes a stream enqueues its work on
 * that stream and returns without waiting for it (sync, size, last_unique,
 * tier_stats and kernel_time wait).  The library launches
 * its kernels with programmatic dependent launch, so a kernel may start while
 * the one before it drains, but each waits for the work before it on entry:
 * stream order holds as for any launch, for the caller's work too.  Calls on one table must
 * be ordered by the caller (one stream, or events between streams).  On an
 * HBM-resident table a sequence of calls can be captured into a CUDA graph and
 * the graph replayed (the same pointers and sizes each replay; the work of
 * each call is device-driven: counts, misses and runs are found on the GPU).
 * Capturing a tiered table's calls returns MLKV_ERR_UNSUPPORTED (its
 * look-ahead runs on the table's own stream).
 *
 * Stale-synchronous mode (staleness_bound s >= 1, the bounded staleness of
 * MLKV Section 3.3.1): issue the gradient applies on one stream and every
 * other call on another.  A Get then waits only for the applies issued more
 * than s applies before it, so it may run while the last s are in flight, and
 * each element it returns holds the effect of every earlier apply except, in
 * any mix, those of the last s (an element is read whole; a row may mix).  In
 * asynchronous mode (MLKV_STALENESS_ASYNC) a Get waits for no apply.  An
 * apply waits for the call issued before it on the other stream (the Get of
 * its keys) and for the apply before it; it inserts no key (an absent key is
 * skipped and MLKV_ERR_NOT_FOUND recorded).  Every other call waits for every
 * apply issued before it (mlkv_dump_keys reads only the index, which applies
 * do not change).  Rows and state after the applies are what
 * bulk-synchronous calls give.  Such a table's calls cannot be captured into a
 * graph (MLKV_ERR_UNSUPPORTED). */

/* Creates a table on the current CUDA device.  Allocates rows + state
 * (capacity x 2 x dim fp32, rows padded to 32 bytes), the index (a power of
 * two >= 2 x capacity slots of 16 bytes) and scratch for max_batch.  With
 * hbm_cache_rows > 0 the rows + state are allocated in host memory instead
 * (capacity slots of pinned host memory from the driver's virtual-memory API,
 * cuMemCreate on the host NUMA node nearest the GPU in 1 GiB chunks, mapped for
 * this device only; the CPU never touches it), with an HBM cache of
 * hbm_cache_rows rows, a row -> location map (cache line or host slot; a row
 * fetched into the cache hands its host slot to the row it evicts), and a side
 * stream for look-ahead.
 * Returns MLKV_ERR_INVALID (bad field), MLKV_ERR_UNSUPPORTED
 * (staleness_bound non-zero with hbm_cache_rows > 0),
 * MLKV_ERR_NOMEM or MLKV_ERR_CUDA.  On success *out
 * owns everything; free it with mlkv_close. */
int mlkv_open(const mlkv_config* cfg, mlkv_table** out);

/* Waits for the table's work, frees all its memory.  Null is a no-op. */
int mlkv_close(mlkv_table* t);

/* Get of MLKV Section 3.1: d_out[i][:] = row of d_keys[i] for i < n.
 * Absent keys: inserted (init row, state_init; row ids handed out in
 * first-occurrence order) when insert_on_miss, otherwise d_out[i][:] = NaN and
 * MLKV_ERR_NOT_FOUND is recorded.  d_out is fp32 [n][dim], 16-byte aligned
 * when dim % 4 == 0. */
int mlkv_get(mlkv_table* t, const int64_t* d_keys, int64_t n, float* d_out, void* stream);

/* Put of MLKV Section 3.1 (upsert): row of d_keys[i] = d_vals[i][:]; a new key
 * is inserted with state_init; a present key keeps its state.  Duplicate keys:
 * the last occurrence wins. */
int mlkv_put(mlkv_table* t, const int64_t* d_keys, int64_t n, const float* d_vals, void* stream);

/* Inserts the absent keys among d_keys with the init row (preloading a key
 * set); present keys are left alone.  Row ids follow first occurrence. */
int mlkv_insert(mlkv_table* t, const int64_t* d_keys, int64_t n, void* stream);

/* The Rmw of MLKV Section 3.2 step 8 with Adagrad: for every distinct key k of
 * d_keys, g = sum of d_grads[i][:] over the i with d_keys[i] == k, then one
 * Adagrad step on k's row and state.  d_grads is fp32 [n][dim].  Absent keys
 * are inserted first when insert_on_miss, else skipped with
 * MLKV_ERR_NOT_FOUND recorded.
 * Tiered table with a look-ahead in flight: this call runs beside the
 * look-ahead (they overlap on the GPU); it may then only update keys that the
 * Get before the look-ahead returned (the training-loop order Get(t),
 * Lookahead(t+1), apply(t)); other keys are skipped with MLKV_ERR_INVALID
 * (absent ones with MLKV_ERR_NOT_FOUND) recorded. */
int mlkv_apply_grad(mlkv_table* t, const int64_t* d_keys, int64_t n, const float* d_grads,
                    void* stream);

/* Lookahead of MLKV Section 3.1 / 3.3.2 with dest = the store's buffer: the
 * rows of d_keys are brought into the HBM cache ahead of use.  A row already
 * resident is not copied again (Section 3.3.2).  With the whole table in HBM
 * every row is resident, so the call checks its arguments and returns.  On a
 * tiered table the work (probe, cache-line hand-out, host <-> HBM swap of
 * each fetched row with the row it evicts) runs on the table's side stream after everything issued
 * on `stream` before it; it does not wait for, and may overlap, the next
 * apply_grad; every other later call waits for it.  Absent keys are skipped
 * (not inserted).  d_keys must stay valid until the look-ahead completes.
 * (dest = the application's cache is a Get into a buffer ahead of use.) */
int mlkv_lookahead(mlkv_table* t, const int64_t* d_keys, int64_t n, void* stream);

/* Checkpoints.  MLKV keeps a store's data by periodic checkpoints (Section
 * 2.2); a checkpoint here is every key in row order (mlkv_dump_keys) with its
 * row and state (mlkv_export), and a restore imports them in that order
 * (mlkv_import), which gives the restored table the same row ids, so training
 * continues bit-identically.
 *
 * mlkv_import: upsert of row and state.  d_rows: fp32 [n][dim]; d_state: fp32
 * [n][dim] or null (a present key keeps its state, a new key gets
 * state_init).  Duplicate keys: the last occurrence wins.  New keys get rows
 * in first-occurrence order, as with insert. */
int mlkv_import(mlkv_table* t, const int64_t* d_keys, int64_t n, const float* d_rows, const float* d_state,
                void* stream);

/* d_keys_out[r] = the key of row r for r < n_rows (n_rows <= mlkv_size(t)):
 * the table's keys in row order.  d_keys_out: device int64 [n_rows]. */
int mlkv_dump_keys(mlkv_table* t, int64_t* d_keys_out, int64_t n_rows, void* stream);

/* Key -> row id (int64, -1 when absent); never inserts. */
int mlkv_find(mlkv_table* t, const int64_t* d_keys, int64_t n, int64_t* d_rows, void* stream);

/* Copies row and state of each key to d_rows / d_state (fp32 [n][dim] each;
 * either may be null); NaN for absent keys.  Never inserts. */
int mlkv_export(mlkv_table* t, const int64_t* d_keys, int64_t n, float* d_rows, float* d_state,
                void* stream);

/* The dedup step of the gradient apply, exposed for checking: the distinct
 * present keys of d_keys ordered by row id, with their occurrence counts.
 * Absent keys are left out and never inserted.  d_unique_keys: int64 [n];
 * d_counts: int32 [n]; *d_num_unique (device int64) = number of distinct
 * present keys. */
int mlkv_dedup(mlkv_table* t, const int64_t* d_keys, int64_t n, int64_t* d_unique_keys,
               int32_t* d_counts, int64_t* d_num_unique, void* stream);

/* Dedup of a batch of raw keys that allocates nothing.  The paper has no
 * counterpart; it is here for callers that must not allocate device memory
 * when they need a dedup: plugins running inside an engine that has reserved
 * the device's memory up front and owns every allocation (a cudaMalloc of
 * theirs can fail, or go behind the engine's accounting), and latency-bound
 * loops where cudaMalloc / cudaFree are banned because they may synchronise
 * the device and stall every stream.  It needs no table.
 *   d_keys: int64 [n], n <= MLKV_STATIC_MAX_KEYS (larger n: MLKV_ERR_INVALID,
 *   nothing enqueued).  Output: the distinct keys in ascending unsigned order
 *   in d_unique_keys (int64 [n]), their occurrence counts in d_counts
 *   (int32 [n]) and their number in *d_num_unique (device int64).  Every key
 *   value is allowed, -1 included.
 * Its working memory is one fixed array in the library's device image (about
 * 1.3 MB, held by every GPU that loads the library until the process exits),
 * so no call allocates.  The first call on a device looks up that array's
 * device address (cudaGetSymbolAddress, with that device current); make that
 * first call before any stream capture.  Every call shares the array: calls
 * that overlap on the GPU (other streams, other host threads) race and give
 * wrong results; order them.  Call with the device of `stream` current. */
#define MLKV_STATIC_MAX_KEYS 65536
int mlkv_dedup_keys_static(const int64_t* d_keys, int64_t n, int64_t* d_unique_keys,
                           int32_t* d_counts, int64_t* d_num_unique, void* stream);

/* Host-buffer forms of Get and the gradient apply: the keys (and gradients)
 * are copied host -> device into table-owned staging on `stream`, the device
 * call runs, and Get's output is copied back to h_out.  The first call
 * allocates the staging (max_batch keys + max_batch x dim floats; on a
 * stale-synchronous table the applies' own second set, so that a Get and an
 * apply on the two streams do not share it).  The call
 * returns once the work is enqueued; h_out is valid after the stream syncs. */
int mlkv_get_host(mlkv_table* t, const int64_t* h_keys, int64_t n, float* h_out, void* stream);
int mlkv_apply_grad_host(mlkv_table* t, const int64_t* h_keys, int64_t n, const float* h_grads,
                         void* stream);

/* Waits for the last stream the table was used on; returns the sticky device
 * status (MLKV_OK when none) or MLKV_ERR_CUDA. */
int mlkv_sync(mlkv_table* t);

/* Clears the sticky device status (synchronises first), and puts back to idle
 * what a call that a device error cut short may have left half done (keys
 * being inserted get no row; a later call inserts them afresh). */
int mlkv_clear_status(mlkv_table* t);

/* Number of distinct keys stored (synchronises). -1 on a null table. */
int64_t mlkv_size(mlkv_table* t);

/* Number of kernels this table has launched since open (host counter). */
int64_t mlkv_launch_count(mlkv_table* t);

/* Tiered table, since open (synchronises; zeros for an HBM-resident table):
 * rows copied host -> HBM cache, rows written back HBM -> host (every evicted
 * row), and cache lines the clock sweep looked at to find victims. */
int mlkv_tier_stats(mlkv_table* t, int64_t* rows_fetched, int64_t* rows_written_back, int64_t* sweep_lines);

/* Per-kernel timing with CUDA events recorded on the launching stream around
 * every launch of kernel `kernel_id` (MLKV_K_*); 0 turns it off.  Read it with
 * mlkv_kernel_time, which synchronises and returns the summed milliseconds and
 * the number of timed launches since the last reset.  While it is on, a
 * gradient apply launches its reduce kernels one after another on the call's
 * stream (otherwise they run on three streams at once), so that each timed
 * launch's events bracket that kernel alone. */
#define MLKV_K_GET_GATHER 1
#define MLKV_K_PROBE 2
#define MLKV_K_SORT_SCATTER 3
#define MLKV_K_REDUCE_SHORT 4
#define MLKV_K_REDUCE_LONG 5
#define MLKV_K_SEGMENTS 6
#define MLKV_K_LONG_COMBINE 7
#define MLKV_K_TIER_FETCH 8
#define MLKV_K_PUT_SCATTER 9
#define MLKV_K_REDUCE_SINGLE 10
#define MLKV_K_REDUCE_SMALL 11
int mlkv_time_kernel(mlkv_table* t, int32_t kernel_id);
int mlkv_kernel_time(mlkv_table* t, double* total_ms, int64_t* launches);

/* Distinct keys of the last gradient apply or dedup (synchronises). */
int64_t mlkv_last_unique(mlkv_table* t);

/* Host-side fault injection, for testing the error paths.  The paper has no
 * counterpart (failure handling is not discussed there).  After
 * mlkv_debug_fail(kind, nth), the nth operation of that kind the library
 * attempts from then on (counting from 1, in any table or in mlkv_open) fails
 * on the host without calling CUDA: for MLKV_FAULT_ALLOC a device or pinned
 * host allocation (cudaMalloc, cudaHostAlloc, a host-tier chunk), which then
 * returns MLKV_ERR_NOMEM; for MLKV_FAULT_COPY a host <-> device copy of a
 * *_host call, which then returns MLKV_ERR_CUDA with nothing after it
 * enqueued; for MLKV_FAULT_WAIT a launch of the kernel that gives new keys
 * their rows (launched by every call that may insert), whose grid barriers then wait for one
 * block more than the grid has: if the call has new keys, every wait runs out
 * (in a second or two), MLKV_ERR_TIMEOUT is recorded and the keys get no rows
 * (a gradient apply still updates the keys that had rows, as if the new keys'
 * lookups were not in the batch; mlkv_clear_status then makes the table whole
 * again).  nth = 0 disarms.  One countdown per kind, shared by the whole
 * process.  No GPU work is affected: nothing faults on the device.  A failed
 * mlkv_open frees everything it allocated and leaves *out null; a failed
 * *_host call leaves the table usable.  Returns MLKV_ERR_INVALID for an
 * unknown kind or nth < 0. */
#define MLKV_FAULT_ALLOC 1
#define MLKV_FAULT_COPY 2
#define MLKV_FAULT_WAIT 3
int mlkv_debug_fail(int32_t kind, int64_t nth);

/* Text of the last error this handle saw (static storage of the handle). */
const char* mlkv_last_error(mlkv_table* t);

/* Text of a status code. */
const char* mlkv_status_string(int status);

#ifdef __cplusplus
}
#endif

#endif /* MLKV_GPU_H */
