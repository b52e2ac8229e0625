/*
 * adapm.h -- C ABI of a GB300 parameter manager driven by intent signals.
 *
 * Method: AdaPM, "Good Intentions: Adaptive Parameter Management via Intent
 * Signaling" (arXiv 2206.00470).  Workers announce, through Intent(), which
 * keys they will access in a window of their own logical clock (Sec. 3).  The
 * manager keeps a replica of each such key at the worker for exactly the
 * span of the intent (Sec. 4.1, selective replication; by default for every
 * active intent, the paper's "AdaPM w/o relocation" of Sec. 5.5, or with
 * relocation when one worker alone has active intent, see adapm_create),
 * serves the worker's reads from the replica, accumulates the worker's writes
 * in it, and merges the accumulated updates into the main copy when the
 * replica is destroyed or when sync() runs (App. B.1.2).  Access without intent is
 * allowed at any time and goes to the main copy (Sec. 4, "optional intent").
 * W workers are worker slots that share one GPU.
 *
 * Conventions for every call
 *   - Keys are uint32 in [0, num_keys).  Value rows are value_len fp32,
 *     row-major, value_len a multiple of 4 (16-byte rows).
 *   - Array arguments may be device pointers or host pointers (pinned or
 *     pageable); the library detects which with cudaPointerGetAttributes.
 *     Host inputs are copied to the device before the call's kernels (pinned
 *     ones on a copy stream of the library's, so that the copy overlaps the
 *     kernels of earlier calls; the library stream waits for it); a host
 *     output is filled by a device-to-host copy on the library stream.
 *   - Calls are ordered on the library stream and return once their work is
 *     enqueued.  Device and pinned host arrays are read and written in
 *     stream order: keep inputs unchanged, and read outputs only, after
 *     adapm_wait() (or a synchronisation of the stream).  Pageable host
 *     inputs are copied before the call returns and may be reused at once.
 *   - The caller owns every array it passes; the library owns all of its
 *     device state and frees it in adapm_destroy().
 *   - Argument errors (null context or pointer, worker >= num_workers,
 *     n > 2^31) return ADAPM_EINVAL synchronously and change nothing.
 *   - Errors found on the device are sticky and returned by adapm_wait():
 *     ADAPM_ERANGE for a key >= num_keys (the element is skipped; a pulled
 *     row for it is zero), ADAPM_ENOMEM when replica_capacity is exhausted
 *     (the replicas of that call are not created and reads of those keys go
 *     to the main copy), ADAPM_ESTATE for a refcount overflow (more than
 *     65535 overlapping intents of one worker on one key).  ADAPM_ETIMEOUT
 *     reports that a bounded device-side wait gave up: the key sort of a
 *     push runs as one cooperative launch whose blocks meet at grid
 *     barriers, and a barrier wait is limited.  Work enqueued after such a failure does not
 *     touch the store, and the context is unusable afterwards (destroy it).
 *   - ADAPM_ECUDA reports a CUDA runtime error; the context is then unusable.
 *   - No C++ exception crosses the ABI.  A context is driven by one host
 *     thread at a time.
 */
#ifndef ADAPM_H
#define ADAPM_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  ADAPM_OK = 0,
  ADAPM_EINVAL = 1,
  ADAPM_ERANGE = 2,
  ADAPM_ENOMEM = 3,
  ADAPM_ESTATE = 4,
  ADAPM_ECUDA = 5,
  ADAPM_ETIMEOUT = 6
} adapm_status;

typedef struct adapm_ctx adapm_ctx; /* opaque; created and freed by the library */

typedef struct {
  uint64_t num_keys;         /* K, 1 <= K < 2^32 - 1 */
  uint32_t value_len;        /* D floats per key, multiple of 4, <= 1024 */
  uint32_t num_workers;      /* W, 1 <= W <= 32 */
  uint64_t replica_capacity; /* max live replicas over all workers; 0 = min(W*K, 2^24) */
  const float* init_values;  /* K*D floats (host or device), copied at create; NULL = zeros */
  void* stream;              /* cudaStream_t to run on; NULL = a stream owned by the library */
  int32_t relocate;          /* 0: replicate every active intent (AdaPM without relocation,
                                Sec. 5.5); 1: relocate a key to the only worker with active
                                intent, replicate while several have it (Sec. 4.1, App. B.2.4) */
  int32_t action_timing;     /* when the manager acts on an intent: ADAPM_ACT_AT_START (0),
                                ADAPM_ACT_ADAPTIVE (1) or ADAPM_ACT_ON_SIGNAL (2), below */
  double timing_alpha;       /* ADAPM_ACT_ADAPTIVE: smoothing factor, 0 = 0.1 */
  double timing_p;           /* ADAPM_ACT_ADAPTIVE: Poisson quantile, 0 = 0.9999 */
  double timing_lambda0;     /* ADAPM_ACT_ADAPTIVE: initial clocks per round, 0 = 10 */
  int32_t delta_refresh;     /* 0: sync refreshes every replica; 1: versioned refresh (see
                                adapm_sync) */
  int32_t no_push_plans;     /* 0: push plans (see adapm_intent) are made and used; 1: never */
  int32_t pull_staging;      /* adapm_pull moves rows 0: through registers (128-bit loads and
                                streaming stores); 1: through shared memory by the bulk-copy
                                engine (1-D cp.async.bulk per row, one bulk store per tile of
                                output rows; used when out is 16-byte aligned) */
  int32_t no_early_events;   /* 0: a worker's next advance computes its refcount events early,
                                beside the worker's pull and push (see adapm_advance_clock);
                                1: never */
} adapm_config;

/* Action timing (Sec. 4.2).
 *   ADAPM_ACT_AT_START   act when the intent becomes active (C^w reaches C_start).
 *   ADAPM_ACT_ON_SIGNAL  act when the intent is signalled: the window is
 *                        treated as starting at the worker's current clock
 *                        (the immediate-action variant of Sec. 5.8).
 *   ADAPM_ACT_ADAPTIVE   Algorithm 1: every adapm_sync is a communication
 *                        round.  After its merge, for each worker w in
 *                        ascending order, with Delta = C^w - (C^w at the
 *                        previous round, 0 at first), the estimate becomes
 *                        (1 - alpha) est + alpha Delta when Delta > 0, and
 *                        every recorded intent of w with
 *                        C^w < C_start < C^w + Q(2 max(est, Delta), p)
 *                        is treated as active from now on (Q = the Poisson
 *                        quantile of adapm_poisson_quantile).  An intent no
 *                        round selected becomes active at C_start.
 * Acting early only moves the start of an intent's window; its end stays. */
#define ADAPM_ACT_AT_START 0
#define ADAPM_ACT_ADAPTIVE 1
#define ADAPM_ACT_ON_SIGNAL 2

/* Create a manager: main store = init_values, every clock 0, no intents, no
 * replicas, every key at its home (owned by no worker).  Memory: K*D*4 (main)
 * + W*K*8 (slot maps, refcounts) + K*8 (holder masks, intent stamps) + K*2
 * with relocate (owner and active-worker count) + K with delta_refresh
 * (written-since-sync flags) + capacity*(2*D*4 + 12)
 * bytes of device memory.  Returns ADAPM_ENOMEM if it does not fit.
 *
 * Relocation (relocate = 1).  Every key has an owner: its home at first,
 * later the last worker that was the only one with active intent for it.
 * The owner reads and writes the main copy directly and holds no replica;
 * every other worker with active intent holds a replica.  Whenever exactly
 * one worker has active intent for a key and does not own it, the key is
 * relocated to that worker: a replica it holds is destroyed first (its
 * pending updates merged into main), then it becomes the owner.  Ownership
 * stays put when the owner's intent expires while others still have active
 * intent (Fig. 10a), and while nobody has.  Pull, push and sync are the
 * same in both modes: a worker without a replica uses the main copy. */
adapm_status adapm_create(const adapm_config* cfg, adapm_ctx** out);

/* Wait for outstanding work and free everything the context owns. */
adapm_status adapm_destroy(adapm_ctx* ctx);

/* Intent(keys, clock_start, clock_end) of `worker` (Sec. 3): the worker will
 * access `keys` while clock_start <= C^worker < clock_end.  Keys are a set:
 * repeats count once.  The optional intent type of the paper is not needed:
 * all types are treated alike (Sec. 4.1).  An empty window (clock_end <=
 * clock_start) or an expired one (clock_end <= C^worker) is a no-op.  A
 * window that contains the current clock is active at once: missing
 * replicas are created before the call's work ends.  Otherwise the keys are
 * de-duplicated and stored until the worker's clock reaches clock_start.
 * Overlapping intents are reference-counted per (worker, key).
 *
 * Push plans (unless no_push_plans).  An intent names the keys a worker
 * will push, before it pushes them (a data loader signals a batch's keys
 * when it builds the batch).  So the call also sorts its keys, with their
 * positions, on a stream of the library's own that runs beside the library
 * stream at low priority; the de-duplicated keys of a window that opens two
 * or more clocks ahead come from that sort.  A push (or training step) of the worker with as many keys
 * as its newest intent whose window holds the current clock checks on the
 * device that its keys equal that intent's, position by position, and then
 * groups its rows by the stored sort instead of sorting again; otherwise it
 * sorts.  Results are the same either way (the same stable order).  The SGNS
 * step, whose rows never follow an intent's key order, always sorts.  A
 * worker whose last four plans went unused gets plans for one intent in
 * sixteen only, until a push takes one again.
 * adapm_wait also waits for that stream. */
adapm_status adapm_intent(adapm_ctx* ctx, uint32_t worker, const uint32_t* keys, uint64_t n,
                          int64_t clock_start, int64_t clock_end);

/* advanceClock() of `worker` (Sec. 3): C^worker += 1.  Replicas whose last
 * active intent expired are destroyed (their updates merged into main), then
 * replicas for keys whose first intent became active are created (value
 * copied from main).  A key that stays active keeps its replica untouched.
 * With relocation, keys are relocated as the worker's intents start and end
 * (see adapm_create); this can destroy another worker's replica.
 *
 * Early events (unless no_early_events; not with relocation or adaptive
 * timing).  The refcount changes of the worker's next advance (which keys
 * gain their first active intent, which lose their last) depend only on the
 * worker's own intents.  So the worker's first adapm_pull, adapm_push or
 * training step after an advance computes them for the intents recorded by
 * then, on a stream of the library's own beside the library stream, and the
 * advance only moves the rows.  If the advance's intents differ from those
 * (one recorded or applied in between), the early changes are undone first.
 * Results are the same either way; adapm_refcounts reports the counts of
 * the worker's current clock.  adapm_wait also waits for that stream. */
adapm_status adapm_advance_clock(adapm_ctx* ctx, uint32_t worker);

/* Read n rows: out[i] = worker's replica of keys[i] if it holds one, else the
 * main copy (Sec. 5.1: reads without replica are current).  Keys may repeat.
 * out: n*D floats, row i for keys[i]. */
adapm_status adapm_pull(adapm_ctx* ctx, uint32_t worker, const uint32_t* keys, uint64_t n,
                        float* out);

/* Write n delta rows: the rows of each distinct key are summed and the sum is
 * added to the worker's replica (its value and its pending-update
 * accumulator) or, without a replica, to the main copy (Sec. 4, App. B.1.2).
 * deltas: n*D floats, row i for keys[i] (a device array that is not 16-byte
 * aligned is first copied to an aligned buffer).  Summation: rows in order of
 * appearance within fixed chunks of the key-sorted batch, chunk sums in
 * chunk order; deterministic for a given input. */
adapm_status adapm_push(adapm_ctx* ctx, uint32_t worker, const uint32_t* keys, uint64_t n,
                        const float* deltas);

/* adapm_push without allocation.  The paper has no counterpart: this entry
 * exists for callers that cannot let the library allocate device memory
 * during a call -- a framework whose own allocator owns the memory budget,
 * or a latency-critical loop in which cudaMalloc/cudaFree may synchronise
 * the device.  Same result as adapm_push (same kernels and summation
 * order), but its scratch is one file-scope device array of 16 MiB that
 * every GPU which loads the library holds until the process exits.
 *   - keys and deltas must be device arrays, deltas 16-byte aligned
 *     (ADAPM_EINVAL otherwise).
 *   - A push whose sort and partial-sum buffers exceed the 16 MiB returns
 *     ADAPM_EINVAL with the sizes in adapm_last_error().  On a 152-SM GPU
 *     every n up to about 790k rows fits at value_len 64, 800k at 200 and
 *     300, 770k at 512 and 710k at 1024.
 *   - The first call on a device looks up the array's device address with
 *     cudaGetSymbolAddress; make that first call before any stream capture.
 *   - Every call (all contexts of the process) shares the one array: calls
 *     that overlap on the GPU (different streams, different contexts) race.
 *   - It allocates nothing: no cudaMalloc, cudaFree or pool allocation.
 *   - Errors and profiling as adapm_push: a CUDA error returns ADAPM_ECUDA
 *     and leaves the context unusable; with adapm_profile_enable on, its
 *     time is recorded under operations 3 (push) and 6 (scatter kernels). */
adapm_status adapm_push_noalloc(adapm_ctx* ctx, uint32_t worker, const uint32_t* keys, uint64_t n,
                                const float* deltas);

/* Replica synchronisation (App. B.1.2): for every key with replicas,
 * main += the pending updates of all holders (ascending worker order), then
 * every holder's replica := main and its pending updates := 0.  With
 * delta_refresh = 1 (App. B.1.2: holders receive only the updates they have
 * not seen) the value of a key's only replica is left as it is when nobody
 * else wrote the key since its last sync (no write to main by a worker
 * without a replica, no destroyed replica): that holder has every update
 * already, its own, so only its pending updates are merged and cleared.
 * Exact arithmetic gives the same values; in fp32 the holder keeps its own
 * rounding of the same sum.  With ADAPM_ACT_ADAPTIVE a sync is also a
 * communication round of Algorithm 1 (see adapm_config), which may activate
 * intents early. */
adapm_status adapm_sync(adapm_ctx* ctx);

/* Block until the stream is idle; return and clear the first sticky device
 * error (ADAPM_ERANGE, ADAPM_ENOMEM, ADAPM_ESTATE) or ADAPM_OK. */
adapm_status adapm_wait(adapm_ctx* ctx);

/* ---- fused training steps (App. C tasks) ------------------------------ */
/* Each reads the rows it needs from the worker's replicas or the main copy
 * (as adapm_pull), computes the loss and gradients of every sample from those
 * values, and pushes one delta row per row occurrence (as adapm_push).  With
 * AdaGrad the value row is [theta | a] (D = 2*dim) and a delta row is
 * [-lr*g/sqrt(a+g*g+eps) | g*g]; without, D = dim and the delta is -lr*g.
 * loss_out (host or device double, may be NULL) receives the batch loss sum,
 * valid after adapm_wait(). */

/* Matrix factorisation, loss 1/2 (v - u.w)^2 per cell (App. C "Matrix
 * factorization"): row_keys[i], col_keys[i], vals[i] for i < n. */
adapm_status adapm_mf_step(adapm_ctx* ctx, uint32_t worker, const uint32_t* row_keys,
                           const uint32_t* col_keys, const float* vals, uint64_t n,
                           uint32_t dim, int adagrad, float lr, float eps, double* loss_out);

/* ComplEx knowledge-graph embeddings with logistic loss (App. C "Knowledge
 * graph embeddings"): rows [re(dim/2) | im(dim/2)] (+ AdaGrad), score
 * Re(sum h r conj(t)); per triple i: heads[i], rels[i], tails[i] positive and
 * neg_tails[i*n_neg + j] negative (label -1).  AdaGrad always (D = 2*dim). */
adapm_status adapm_complex_step(adapm_ctx* ctx, uint32_t worker, const uint32_t* heads,
                                const uint32_t* rels, const uint32_t* tails,
                                const uint32_t* neg_tails, uint64_t n, uint32_t n_neg,
                                uint32_t dim, float lr, float eps, double* loss_out);

/* Skip-gram with negative sampling, plain SGD (App. C "Word vectors"): input
 * vector of token c is key c, output vector of token o is key vocab + o.
 * centres[i]; contexts[i*n_ctx + j] (0xFFFFFFFF = no context in that slot);
 * negatives[(i*n_ctx + j)*n_neg + q].  D = dim. */
adapm_status adapm_sgns_step(adapm_ctx* ctx, uint32_t worker, const uint32_t* centres,
                             const uint32_t* contexts, const uint32_t* negatives, uint64_t n,
                             uint32_t n_ctx, uint32_t n_neg, uint32_t vocab, uint32_t dim,
                             float lr, double* loss_out);

/* ---- inspection (synchronising; for tests and tools) ------------------ */
adapm_status adapm_clock(adapm_ctx* ctx, uint32_t worker, int64_t* out);

/* Keys of the worker's replicas in ascending order: the logical slot map
 * (slot of key k = rank of k in this list).  Writes min(cap, count) keys to
 * out (host or device) and the count to *n (host). */
adapm_status adapm_replica_keys(adapm_ctx* ctx, uint32_t worker, uint32_t* out, uint64_t cap,
                                uint64_t* n);

/* For each key: has[i] = 1 if the worker holds a replica, and its value row
 * and pending-update row (zeros when it holds none). */
adapm_status adapm_replica_rows(adapm_ctx* ctx, uint32_t worker, const uint32_t* keys, uint64_t n,
                                float* val_out, float* acc_out, uint8_t* has_out);

/* Number of the worker's active intents containing each key (uint32 out). */
adapm_status adapm_refcounts(adapm_ctx* ctx, uint32_t worker, const uint32_t* keys, uint64_t n,
                             uint32_t* out);

/* The p quantile of a Poisson distribution with mean lambda: the smallest
 * integer q >= 0 with P(X <= q) >= p, found by adding P(X = j) =
 * exp(-lambda + j ln lambda - ln j!) for j = 0, 1, ... in that order (the
 * rule ADAPM_ACT_ADAPTIVE uses).  Host only; needs no GPU.  ADAPM_EINVAL
 * unless lambda > 0, 0 < p < 1 and out is not NULL. */
adapm_status adapm_poisson_quantile(double lambda, double p, int64_t* out);

/* Owner of each key (int32 out): the worker that holds the key's main copy,
 * -1 while it is at its home.  Always -1 without relocation. */
adapm_status adapm_owners(adapm_ctx* ctx, const uint32_t* keys, uint64_t n, int32_t* out);

/* Rows of the main copy. */
adapm_status adapm_read_main(adapm_ctx* ctx, const uint32_t* keys, uint64_t n, float* out);

typedef struct {
  uint64_t live_replicas;    /* replicas that exist now, all workers */
  uint64_t high_water;       /* replica slots ever in use */
  uint64_t capacity;
  uint64_t created, destroyed;
  uint64_t last_push_unique; /* distinct keys of the last push */
  uint64_t push_rows;        /* rows pushed, cumulative (training steps included) */
  uint64_t push_unique;      /* distinct keys per push, summed over pushes */
  uint64_t sync_keys;        /* keys merged by sync, cumulative */
  uint64_t sync_replicas;    /* replicas refreshed by sync, cumulative */
  uint64_t relocations;      /* owner changes, cumulative (relocation only) */
  uint64_t sync_refreshed;   /* replica values written by sync, cumulative */
  uint64_t planned_pushes;   /* pushes that checked a push plan (see adapm_intent), cumulative */
  uint64_t plan_misses;      /* of those, pushes whose keys differed, so they sorted, cumulative */
  uint64_t early_advances;   /* advances whose refcount events ran early, cumulative */
  uint64_t early_undone;     /* early events undone (the advance's intents changed), cumulative */
} adapm_stats;

adapm_status adapm_get_stats(adapm_ctx* ctx, adapm_stats* out);

/* Per-operation device time: when enabled, every call records CUDA events
 * around its work on the library stream.  Operations: 0 intent, 1 advance,
 * 2 pull, 3 push, 4 sync, 5 training-step compute (without its push),
 * 6 push gather-scatter kernel alone, 7 pull gather kernel alone.
 * adapm_profile_read synchronises and returns the summed milliseconds and
 * call counts since the last read (arrays of ADAPM_NUM_OPS). */
#define ADAPM_NUM_OPS 8
adapm_status adapm_profile_enable(adapm_ctx* ctx, int enable);
adapm_status adapm_profile_read(adapm_ctx* ctx, double* ms_out, uint64_t* calls_out);

/* Number of CUDA kernels this library has launched in this process (all
 * contexts), for checking which work ran on the GPU. */
adapm_status adapm_kernel_launches(uint64_t* out);

/* Message for the last error returned on this context ("" if none). */
const char* adapm_last_error(adapm_ctx* ctx);

/* Fault injection for tests of the bounded device waits (no GPU fault is
 * involved): the next push of this context sorts its keys in a launch whose
 * first grid barrier waits for arrivals that never come.  That wait gives up
 * after about a second, the push leaves the store untouched, and
 * adapm_wait returns ADAPM_ETIMEOUT; the context is unusable afterwards,
 * other contexts are unaffected. */
adapm_status adapm_debug_fail_next_barrier(adapm_ctx* ctx);

/* Fault injection for tests of CUDA error handling (no GPU fault is
 * involved, nothing on the device changes): the next call of this context
 * that launches kernels enqueues them and then returns ADAPM_ECUDA as if
 * the CUDA runtime had reported a launch failure.  As after a real one, the
 * context is unusable afterwards (every later call returns ADAPM_ECUDA);
 * other contexts are unaffected. */
adapm_status adapm_debug_fail_next_launch(adapm_ctx* ctx);

#ifdef __cplusplus
}
#endif
#endif /* ADAPM_H */
