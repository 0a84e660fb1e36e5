/*
 * dualmap.h -- C ABI of a GB300 (sm_103a) implementation of DualMap's batched
 * request-routing path (arxiv 2602.06502, "DualMap: Enabling Both Cache
 * Affinity and Load Balancing for Distributed LLM Serving").
 *
 * One handle is one global scheduler (Sec. 3.1): a cluster of up to
 * `max_instances` inference instances, two consistent-hash rings, a per-
 * instance index of cached prefix blocks, and per-instance FIFO queues of
 * pending prefill work.  All state lives in device memory owned by the
 * handle.  Work is enqueued on the handle's CUDA stream; calls return as soon
 * as the work is enqueued unless stated otherwise.
 *
 * Conventions
 *   - "device" pointers are CUDA device (or managed) memory, "host" pointers
 *     are host memory.  The caller owns every buffer passed in; it must stay
 *     valid until the handle's stream has executed the call.
 *   - Synchronous argument checks return an error and change nothing.
 *   - Checks that need device data (prompt lengths, offsets, capacities) run
 *     in the kernels: a failure is recorded as a sticky device error, the
 *     rest of that call's kernels do nothing, and every later call that
 *     changes state returns the error (see dm_last_error); the read-only
 *     calls (dm_get_loads, dm_export_*, dm_get_clock) keep working.  The
 *     handle must then be destroyed.
 *   - One handle must be used from one host thread at a time.
 *
 * Readings of details the paper leaves open (block size, hash family, ring
 * layout, tie rules, time model) are fixed once here and implemented
 * identically by the independent CPU oracle used in the tests.
 */
#ifndef DUALMAP_H
#define DUALMAP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define DM_API __attribute__((visibility("default")))
#else
#define DM_API
#endif

typedef struct dm_handle dm_handle;

typedef enum {
    DM_OK = 0,
    DM_ERR_INVALID_ARG = 1,   /* bad argument (null pointer, prompt < 1 block, misaligned offset...) */
    DM_ERR_CAPACITY = 2,      /* a max_* bound of dm_config would be exceeded */
    DM_ERR_NO_INSTANCES = 3,  /* routing needs at least two live instances */
    DM_ERR_DUPLICATE_ID = 4,  /* id already live, or removed and still draining */
    DM_ERR_UNKNOWN_ID = 5,    /* id not live */
    DM_ERR_ORDER = 6,         /* batch time earlier than the previous batch's */
    DM_ERR_CUDA = 7,          /* a CUDA runtime call failed */
    DM_ERR_TIMEOUT = 8,       /* a bounded device-side loop gave up (state is corrupt) */
    DM_ERR_OOM = 9,           /* device or host allocation failed */
    DM_ERR_BOUNDS = 10        /* debug builds only (libdualmap_debug.so): a device-side index check failed */
} dm_status;

/* Choice rules of dm_route_batch's last step.
 *
 * DualMap's own rule (Sec. 3.2): ttft_f = W[c_f] + cost * (L - hit_f); the
 * candidate with more hit tokens unless its ttft exceeds the SLO, then the
 * less-loaded (by W) of the two, tie: the higher-hit one ("switched");
 * equal hits take the less-loaded, tie c1.
 *
 * Between the same two candidates (the ablation variants of Sec. 4.3):
 *   PAIR_CACHE_AFFINITY  more hit tokens; equal hits: less loaded, tie c1.
 *   PAIR_LEAST_LOADED    smaller W, tie c1.
 *   PAIR_MIN_TTFT        smaller ttft_f, tie c1.
 *   PAIR_PREBLE          2 * max(hit1, hit2) > L ? PAIR_CACHE_AFFINITY
 *                        : PAIR_MIN_TTFT (Preble's 50% rule, Sec. 2.2).
 *   switched = the hits differ and the candidate with fewer was chosen.
 * Over every live instance (the cluster-wide baselines of Sec. 2.2 and
 * Sec. 4; hit_i is probed on every live instance, an extra kernel whose
 * cost grows with the instance count):
 *   CACHE_AFFINITY  always c1, the ring-1 owner (one prompt-aware mapping).
 *   LEAST_LOADED    smallest W_i, tie lowest id.
 *   MIN_TTFT        smallest W_i + cost * (L - hit_i), tie lowest id
 *                   (Mooncake's rule as Sec. 2.2 describes it).
 *   PREBLE          2 * max_i hit_i > L ? among the instances with that hit
 *                   the smallest W_i, tie lowest id : MIN_TTFT.
 *   switched = 0; ttft1/ttft2 still describe the two candidates, and the
 *   queued work is cost * (L - hit) of the chosen instance. */
typedef enum {
    DM_RULE_DUALMAP = 0,
    DM_RULE_PAIR_CACHE_AFFINITY = 1,
    DM_RULE_PAIR_LEAST_LOADED = 2,
    DM_RULE_PAIR_MIN_TTFT = 3,
    DM_RULE_PAIR_PREBLE = 4,
    DM_RULE_CACHE_AFFINITY = 5,
    DM_RULE_LEAST_LOADED = 6,
    DM_RULE_MIN_TTFT = 7,
    DM_RULE_PREBLE = 8
} dm_choice_rule;

/* Scheduler configuration (copied at dm_create). */
typedef struct {
    /* Tokens per block, B.  One of 4, 8, 16, 32, 64.  Blocks are the unit of
     * prefix keys and of the cache index (App. A.1.1 uses 512-token hash
     * blocks, App. A.3.2 128-token KV blocks; a single block size serves both
     * here).  Only full blocks are keyed. */
    uint32_t block_tokens;
    /* Blocks hashed into the ring key, K_route in 1..256 (Sec. 3.2 "how long
     * a prefix"); a prompt with fewer full blocks uses all of them. */
    uint32_t route_prefix_blocks;
    /* Virtual nodes per instance on each ring, V >= 1 (Sec. 3.4). */
    uint32_t vnodes_per_instance;
    /* Instance ids are 0 .. max_instances-1; 2 <= max_instances <= 8192. */
    uint32_t max_instances;
    /* Cache index capacity per instance in blocks, C >= 1 (exact LRU). */
    uint64_t cache_capacity_blocks;
    /* TTFT SLO in integer microseconds (Sec. 3.2). */
    uint64_t slo_us;
    /* Prefill cost in integer microseconds per uncached token, >= 1. */
    uint32_t cost_us_per_token;
    /* Hotspot rule of dm_rebalance: instance i is hot when
     * hot_den * N * W_i > hot_num * sum(W) (3/2 = 1.5x the mean). */
    uint32_t hot_num, hot_den;
    /* Largest batch, in requests (>= 1). */
    uint32_t max_batch;
    /* Largest token buffer of a batch (dm_batch.total_tokens), >= B. */
    uint64_t max_batch_tokens;
    /* Largest number of blocks one commit may touch on one instance; 0 means
     * max_batch_tokens / B.  Sizes each instance's index (2 x (C + this),
     * rounded up to a power of two, 16 bytes a slot) and recency log. */
    uint64_t max_touch_per_instance;
    /* Queue capacity per instance in entries (power of two); 0 = 65536. */
    uint32_t max_queue;
    /* log2 of the index slots per instance; 0 = automatic, the smallest
     * power of two >= 2 x (C + max_touch_per_instance).  A larger index is
     * rebuilt less often (it is rebuilt when a quarter full if a quarter
     * still holds C + max_touch_per_instance keys, else when half full,
     * counting the slots evicted keys keep).  Never smaller than the
     * automatic size, nor than 64; <= 32.  dm_create returns DM_ERR_INVALID_ARG when the resulting
     * index would exceed 2^32 slots (it records slot numbers as 32 bits). */
    uint32_t index_slots_log2;
    /* The choice rule of dm_route_batch (dm_choice_rule); 0 = DualMap's
     * SLO-aware rule.  The others are the rules DualMap is compared with,
     * for experiments; DM_ERR_INVALID_ARG for an unknown value.  The
     * cluster-wide rules allocate max_batch x max_instances u32 hit counts
     * (DM_ERR_OOM when that does not fit). */
    uint32_t choice_rule;
    /* Adaptive hash-prefix length (Sec. 3.2, "how long prefix is
     * appropriate"); adapt_step_blocks = 0 keeps every request at
     * min(K_route, n_blk).  Otherwise a prefix hotness tree decides each
     * request's length: a node is a prefix, named by its last block's key;
     * a request starts at min(K_route, n_blk) blocks and, while its node is
     * expanded and its prompt and adapt_max_blocks allow, goes
     * adapt_step_blocks deeper (capped by n_blk and adapt_max_blocks).  Every
     * adapt_window routed non-empty batches form a window; at its end, with
     * n live instances and T requests in the window, a node reached by more
     * than 2T/n of them (and shorter than adapt_max_blocks) is expanded and
     * an expanded node reached by fewer than T/n is dropped; the new tree
     * applies from the next batch.  K_route < adapt_max_blocks <= 2048,
     * adapt_window >= 1, and the window's node-count table (2 x max_batch x
     * adapt_window x levels entries of 16 bytes, levels = ceil((adapt_max_blocks
     * - K_route) / adapt_step_blocks) + 1) at most 2^26 entries;
     * DM_ERR_INVALID_ARG otherwise. */
    uint32_t adapt_step_blocks;
    uint32_t adapt_max_blocks;
    uint32_t adapt_window;
    /* Variants of dm_rebalance (DM_REBALANCE_* bits); 0 = the rule described
     * at dm_rebalance. */
    uint32_t rebalance_flags;
    /* Spare index buffers shared by all instances as rebuild targets (a
     * rebuild builds the new index in a spare and returns the old one to the
     * pool); 0 = one per instance (index memory: two indices per instance).
     * A pool much smaller than max_instances nearly halves the index memory;
     * rebuilds beyond the pool then wait their turn (round robin), so
     * dm_create requires index_slots / 2 >= ceil(max_instances /
     * rebuild_pool) * max_touch_per_instance (DM_ERR_INVALID_ARG otherwise). */
    uint32_t rebuild_pool;
    /* Testing only (no paper counterpart); 0 in normal use.  A nonzero value
     * caps the iterations of the data-dependent device loops of the cache
     * index (bucket walks of a lookup, retries of a touch) at that many, so
     * a test can make a bounded loop give up: the call then records
     * DM_ERR_TIMEOUT as a sticky error, like an exhausted bound in normal
     * use. */
    uint32_t test_loop_limit;
    /* Candidates per request (App. A.8, "Optimal Candidate Set Size"): 0 or 2
     * is DualMap's two (dm_route_batch); 1 or 3..8 routes with that many
     * independent hash functions, rings and probes through dm_route_batch_d
     * (with choice_rule 0 and the fixed prefix length only;
     * DM_ERR_INVALID_ARG otherwise, and dm_route_batch and dm_rebalance
     * return DM_ERR_INVALID_ARG on such a handle). */
    uint32_t candidates;
    /* With DM_REBALANCE_FRESH_HITS: the capacity, in blocks, of each
     * instance's ring of its queued requests' block keys (rounded up to a
     * power of two; device memory: 8 bytes x this x max_instances).  It must
     * hold the keys of every request queued on an instance at once: a
     * routing or rebalance call that would outgrow it records
     * DM_ERR_CAPACITY (sticky).  Required > 0 with that flag
     * (DM_ERR_INVALID_ARG otherwise), ignored without it. */
    uint64_t rebalance_key_blocks;
    /* Seed of all hash key material (SplitMix64). */
    uint64_t seed;
    /* cudaStream_t for all work of this handle; NULL = legacy default stream. */
    void *stream;
} dm_config;

/* One batch of requests in arrival order.
 * Prompt r is tokens[offsets[r] .. offsets[r] + lengths[r]) (uint32 token
 * ids).  For the device entry points `tokens` must be 16-byte aligned
 * (DM_ERR_INVALID_ARG otherwise).  Every offsets[r] must be a multiple of 4
 * (prompts start on 16-byte boundaries) and offsets[r] + lengths[r] <=
 * total_tokens; prompts may overlap or share tokens.  lengths[r] >=
 * block_tokens. */
typedef struct {
    const uint32_t *tokens;     /* device (host for dm_route_batch_host) */
    const uint64_t *offsets;    /* device (host ...), n entries */
    const uint32_t *lengths;    /* device (host ...), n entries */
    uint32_t n;                 /* requests, <= max_batch; 0 = only advance time */
    uint32_t reserved0;         /* must be 0 */
    uint64_t total_tokens;      /* extent of tokens[], <= max_batch_tokens */
    uint64_t batch_time_us;     /* arrival time of the batch's last request */
} dm_batch;

/* Per-request results of dm_route_batch (n entries each, device memory;
 * host memory for dm_route_batch_host). */
typedef struct {
    uint32_t *cand1;     /* first candidate: owner of pos1 on ring 1 */
    uint32_t *cand2;     /* second candidate (distinct from cand1) */
    uint32_t *hit1;      /* cached-prefix tokens on cand1 (multiple of B) */
    uint32_t *hit2;      /* cached-prefix tokens on cand2 */
    uint64_t *ttft1;     /* estimated TTFT on cand1, us */
    uint64_t *ttft2;     /* estimated TTFT on cand2, us */
    uint32_t *chosen;    /* instance the request is queued on */
    uint8_t *switched;   /* 1 when the SLO rule overrode cache affinity */
} dm_route_out;

/* Per-request results of dm_route_batch_d with d candidates (device
 * memory): cand, hit and ttft hold n x d entries, request-major (request r,
 * candidate f at r * d + f, f in ring order 1..d). */
typedef struct {
    uint32_t *cand;      /* the d distinct candidates */
    uint32_t *hit;       /* cached-prefix tokens on each (multiple of B) */
    uint64_t *ttft;      /* estimated TTFT on each, us */
    uint32_t *chosen;    /* instance the request is queued on (n entries) */
    uint8_t *switched;   /* 1 when the SLO rule overrode cache affinity (n entries) */
} dm_route_out_d;

typedef struct {
    uint64_t req_seq;    /* global request sequence number (0-based, arrival order) */
    uint32_t from, to;
} dm_migration;

/* Stages timed by dm_get_stage_times. */
enum {
    DM_STAGE_SETUP = 0,    /* batch validation and per-request prefix sums */
    DM_STAGE_DRAIN = 1,    /* queue draining to the batch time (runs inside the setup
                              stage's kernel, so it is timed there; 0 calls) */
    DM_STAGE_HASH = 2,     /* token hashing into chained block prefix values */
    DM_STAGE_PROBE = 3,    /* ring lookup, distinct fix, cache probes */
    DM_STAGE_CHOICE = 4,   /* sequential choice (with the all-instance probes of the
                              cluster-wide rules) */
    DM_STAGE_COMMIT = 5,   /* cache commit with LRU eviction */
    DM_STAGE_REBALANCE = 6,/* hotspot-aware rebalancing */
    DM_STAGE_COUNT = 7
};

/* dm_config.rebalance_flags.  DM_REBALANCE_SLO_TARGET: an instance is
 * overloaded when its queued work exceeds the SLO, and migration from it
 * stops once its queued work is within the SLO (Sec. 3.3: "until all
 * requests in the overloaded instance's queue are expected to meet the
 * TTFT SLO"), instead of the 1.5x-mean hotspot rule.
 * DM_REBALANCE_DOUBLE_OVERLOAD: dm_rebalance migrates only if, in the last
 * routed batch, some request's estimated TTFT exceeded the SLO on both of
 * its candidates (App. A.1.2: rebalancing starts "whenever both candidate
 * instances of a request are identified as overloaded").
 * DM_REBALANCE_FRESH_HITS: a migration candidate's TTFT on its other
 * candidate uses the cached-prefix length found by probing that instance's
 * index as it stands at the call, with the request's own block keys (kept
 * for every queued request in per-instance rings, see
 * dm_config.rebalance_key_blocks), instead of the length found when it was
 * routed (Sec. 3.3's benefit with a fresh query of the instance's KV
 * metadata).  With the pair rules (choice_rule < 5) and two candidates only
 * (DM_ERR_INVALID_ARG otherwise). */
#define DM_REBALANCE_SLO_TARGET 1u
#define DM_REBALANCE_DOUBLE_OVERLOAD 2u
#define DM_REBALANCE_FRESH_HITS 4u

/* Create a scheduler with no instances (the global scheduler of Sec. 3.1;
 * the paper describes no construction step, so this lifecycle call and
 * dm_destroy cite no passage).  Allocates all device state except the
 * per-instance indices (allocated on first dm_add_instance of an id).
 * Derives the hash key material from cfg->seed.  On success *out owns the
 * handle (release it with dm_destroy); on failure *out is NULL and nothing
 * is left allocated: DM_ERR_INVALID_ARG for a field outside the ranges
 * stated in dm_config, DM_ERR_OOM when device memory runs out, DM_ERR_CUDA
 * for another runtime failure.  Synchronous. */
DM_API dm_status dm_create(const dm_config *cfg, dm_handle **out);

/* Destroy a handle, synchronising its stream first and freeing all its
 * device memory.  NULL is ignored. */
DM_API void dm_destroy(dm_handle *h);

/* Add instance `id` (Sec. 3.4, App. A.1.3): inserts its V virtual nodes into
 * both rings (only keys on its new arcs remap) and gives it an empty index
 * and queue.  DM_ERR_DUPLICATE_ID if it is live, or removed but its queue
 * has not drained yet.  Synchronous (it reads the queue state). */
DM_API dm_status dm_add_instance(dm_handle *h, uint32_t id);

/* Remove instance `id`: deletes its virtual nodes from both rings; its
 * queued work keeps draining, it receives no new requests and no
 * migrations.  DM_ERR_UNKNOWN_ID if not live.  Asynchronous. */
DM_API dm_status dm_remove_instance(dm_handle *h, uint32_t id);

/* Route one batch (Sec. 3.2, App. A.1.1):
 *   1. every queue drains by batch_time_us minus the previous batch time;
 *   2. each prompt is hashed block by block into chained 64-bit prefix
 *      values under two independent hash functions; the first
 *      min(K_route, n_blk) blocks give two ring positions;
 *   3. each position's successor virtual node on its ring gives a candidate;
 *      equal candidates are separated by taking the next live id;
 *   4. each candidate's index is probed for the leading run of resident
 *      block keys (index state as of the start of the batch);
 *   5. in arrival order: TTFT_f = W[c_f] + cost * (L - hit_f); the higher-hit
 *      candidate unless its TTFT exceeds the SLO, then the less-loaded one;
 *      equal hits take the less-loaded one; the request is queued there
 *      (or the configured dm_choice_rule decides).
 * The batch is kept for dm_commit_cache.  Asynchronous. */
DM_API dm_status dm_route_batch(dm_handle *h, const dm_batch *batch, const dm_route_out *out);

/* Route one batch with d candidates instead of two (App. A.8: the paper
 * weighs the candidate set size d and keeps d = 2), d = dm_config.candidates
 * (2 on a handle created with 0 or 2).  Per request: the prompt prefix
 * hashed under d independent functions (functions 1 and 2 are
 * dm_route_batch's; functions 3..d draw their key material from the seed
 * after DualMap's), one position per ring, the successor's owner on each of
 * d rings, made distinct (an owner already taken by an earlier ring is
 * replaced by the next live id after it, in ascending order, cyclically,
 * not yet taken), the leading run of resident blocks on each candidate,
 * then DualMap's rule over d candidates: among the candidates with the most
 * hit tokens, a = the less loaded by W (tie: the earlier ring); a is chosen
 * when every candidate has that many hits or TTFT_a <= SLO; otherwise the
 * least loaded candidate by W (tie: a, then the earlier ring), flagged
 * "switched".  d = 2 gives dm_route_batch's decisions; d = 1 always takes
 * the ring-1 owner (cache affinity).  Time, loads, queues, metrics and the
 * following dm_commit_cache are those of dm_route_batch; queue entries
 * keep the first two candidates.  DM_ERR_NO_INSTANCES with fewer than
 * max(2, d) live instances.  Asynchronous. */
DM_API dm_status dm_route_batch_d(dm_handle *h, const dm_batch *batch, const dm_route_out_d *out);

/* Same as dm_route_batch with every pointer of `batch` and `out` in host
 * memory (pinned memory is faster).  The library copies the inputs to its
 * own device staging buffers, routes, copies the results back and
 * synchronises the stream before returning. */
DM_API dm_status dm_route_batch_host(dm_handle *h, const dm_batch *batch, const dm_route_out *out);

/* Asynchronous dm_route_batch_host: returns once the work is enqueued.  The
 * library alternates between two device staging buffers, uploading a batch
 * on its own copy stream while the previous batch routes, so the caller's
 * host input and output buffers must stay untouched until the handle's
 * stream has been synchronised (dm_last_error does).  Use pinned host memory
 * for the copies to overlap. */
DM_API dm_status dm_route_batch_host_async(dm_handle *h, const dm_batch *batch, const dm_route_out *out);

/* Sharded routing (no paper counterpart: the multi-GPU split of the routing
 * step).  Each of several handles holds the same replicated state (same
 * config and seed, same instance adds/removes, same batches), typically
 * one per GPU.  For a batch of n requests each handle calls
 * dm_route_shard_begin with its own request range [r0, r1) (the ranges
 * partition [0, n)): it drains the queues and lays the whole batch out
 * exactly as dm_route_batch does, but hashes, looks up and probes only
 * requests r0 .. r1-1 (Sec. 3.2, App. A.3.2 for those steps).  It then
 * exports its results with dm_shard_export, the callers exchange the
 * buffers (an all-gather), every handle imports the other ranges with
 * dm_shard_import, and dm_route_shard_finish runs the rest of the step
 * (choices in arrival order, queues, metrics; the batch becomes the pending
 * commit) on the whole batch.  Every handle then holds the outputs and state
 * that dm_route_batch would have produced.  Not with the adaptive prefix
 * length (DM_ERR_INVALID_ARG).  Between begin and finish every other call
 * that routes, commits, rebalances, hashes or changes the instances returns
 * DM_ERR_ORDER.
 *
 * Export buffer (device memory, 8-byte aligned, written in stream order):
 * the local prefix values of the range's blocks (8 bytes each), its
 * segments' f1 totals (8 bytes), then 4-byte values: its segments' owning
 * requests, and per request its hash length, both candidates and both first
 * missing blocks, array by array.  `*bytes_dev` (device, may be null)
 * receives the size: 8 (blocks + segments) + 4 (segments + 5 requests);
 * a buffer smaller than that records DM_ERR_CAPACITY (sticky).  Import reads
 * the same layout for its range from `buf_dev` (`bytes` long). */
DM_API dm_status dm_route_shard_begin(dm_handle *h, const dm_batch *batch, uint32_t r0, uint32_t r1);
DM_API dm_status dm_shard_export(dm_handle *h, uint32_t r0, uint32_t r1, void *buf_dev, uint64_t cap,
                                 uint64_t *bytes_dev);
DM_API dm_status dm_shard_import(dm_handle *h, uint32_t r0, uint32_t r1, const void *buf_dev, uint64_t bytes);
DM_API dm_status dm_route_shard_finish(dm_handle *h, const dm_batch *batch, const dm_route_out *out);

/* Hotspot-aware rebalancing (Sec. 3.3, Eq. "rebalance"; App. A.1.2), to be
 * called after dm_route_batch and before dm_commit_cache.  Hot instances
 * (hot_den * N * W_i > hot_num * sum W, or see DM_REBALANCE_SLO_TARGET)
 * are visited in descending W; their queued, not-started requests are
 * ranked by migration benefit B = TTFT_{r,i} - TTFT_{r,j} (j the request's
 * other candidate) and moved to j while i stays hot, B > 0 and
 * TTFT_{r,j} < SLO.  Writes up to `cap` migrations, in the order they were
 * made, to out_host (host memory, owned by the caller) and the total
 * number made to *n_out (host; it may exceed cap).  Synchronous: the
 * migrations are computed on the device and copied back before it returns
 * (the library keeps a device staging buffer of `cap` entries, grown on
 * demand: DM_ERR_OOM if that fails).  DM_ERR_INVALID_ARG if n_out is NULL,
 * or out_host is NULL with cap > 0. */
DM_API dm_status dm_rebalance(dm_handle *h, dm_migration *out_host, uint32_t cap, uint32_t *n_out);

/* dm_rebalance with device outputs, for a pipeline that keeps the results
 * on the GPU: up to `cap` migrations to out_dev (device) and the total
 * count to *n_out_dev (device), enqueued on the handle's stream.
 * Asynchronous. */
DM_API dm_status dm_rebalance_async(dm_handle *h, dm_migration *out_dev, uint32_t cap, uint32_t *n_out_dev);

/* Cache save (App. A.3.2) of the last routed batch: in arrival order, each
 * request touches its block keys on its final instance (block n_blk-1 down
 * to 0, one global clock tick each); each index then keeps its C most
 * recently touched keys (exact LRU).  A no-op when the last batch is
 * already committed.  Asynchronous. */
DM_API dm_status dm_commit_cache(dm_handle *h);

/* Chained block keys and ring positions of a batch without touching any
 * scheduler state: keys_dev receives, for request r, its n_blk(r) = L/B
 * cache keys at positions key_off[r] .. key_off[r] + n_blk(r), where
 * key_off (device, n+1 entries, written by the call) is the exclusive prefix
 * sum of n_blk; pos_dev (device, 2n entries) receives (pos1, pos2) per
 * request, hashed over min(K_route, n_blk) blocks (the fixed length, also
 * with the adaptive length on).  keys_dev must hold sum(n_blk) entries (at
 * most total_tokens / B).  Asynchronous. */
DM_API dm_status dm_hash_prompts(dm_handle *h, const dm_batch *batch, uint64_t *keys_dev,
                          uint64_t *key_off_dev, uint64_t *pos_dev);

/* Limits of dm_hash_prompts_noalloc: requests per call, and full blocks per
 * call (total_tokens / block_tokens).  Its fixed scratch is about 2.2 MB. */
#define DM_NOALLOC_MAX_REQUESTS 4096u
#define DM_NOALLOC_MAX_BLOCKS 4194304ull

/* dm_hash_prompts without any device allocation, and without a handle: the
 * same block keys, key offsets and ring positions as dm_hash_prompts on a
 * handle created with this block_tokens, route_prefix_blocks and seed.  The
 * paper has no counterpart; it exists for callers that cannot allocate
 * device memory at the point they hash, for example a serving process whose
 * device memory is entirely owned by another allocator, or code on a path
 * where cudaMalloc's implicit synchronisation is not acceptable.
 * Working memory is one fixed array of about 2.2 MB inside the library, which
 * every GPU that loads the library keeps until the process exits; keys_dev
 * (which must hold sum(n_blk) entries) doubles as working space.
 * Returns DM_ERR_CAPACITY without doing anything when n exceeds
 * DM_NOALLOC_MAX_REQUESTS or total_tokens / block_tokens exceeds
 * DM_NOALLOC_MAX_BLOCKS; device-side checks (prompt lengths and offsets, the
 * exact block count) are reported by the return value: every call
 * synchronises `stream` (a cudaStream_t, NULL = legacy default stream) and
 * reads the device error word back before returning, so no call may be made
 * while any stream on that device is capturing.  The first call on each
 * device looks up the array's device address; the address is kept for the life of the
 * process, so after a cudaDeviceReset of a device the entry point must not be
 * called on that device again.  Every call uses the same array: calls whose
 * work overlaps on the GPU (other host threads, other streams) race and
 * produce garbage, so the caller serialises them. */
DM_API dm_status dm_hash_prompts_noalloc(uint32_t block_tokens, uint32_t route_prefix_blocks, uint64_t seed,
                                         const dm_batch *batch, uint64_t *keys_dev, uint64_t *key_off_dev,
                                         uint64_t *pos_dev, void *stream);

/* Raw ring owners (before the distinct fix) of n positions: pos_dev holds
 * (pos1, pos2) pairs as written by dm_hash_prompts; owner1_dev/owner2_dev
 * receive the successor's owner on ring 1 / ring 2.  Asynchronous. */
DM_API dm_status dm_ring_lookup(dm_handle *h, const uint64_t *pos_dev, uint32_t n,
                         uint32_t *owner1_dev, uint32_t *owner2_dev);

/* Queued prefill work W (us) of every instance id (the load of Sec. 3.2):
 * W_host (host, caller-owned) receives ids 0 .. min(cap, max_instances)-1
 * (0 for ids never added), and *n_out (host) the number of ids,
 * max_instances.  DM_ERR_INVALID_ARG if n_out is NULL, or W_host is NULL
 * with cap > 0.  Synchronous; works after a sticky error. */
DM_API dm_status dm_get_loads(dm_handle *h, uint64_t *W_host, uint32_t cap, uint32_t *n_out);

/* Resident (key, last-touch stamp) pairs of instance `id`, in unspecified
 * order; *n_out = resident count (entries beyond cap are not written).
 * Synchronous. */
DM_API dm_status dm_export_cache(dm_handle *h, uint32_t id, uint64_t *keys_host, uint64_t *stamps_host,
                          uint64_t cap, uint64_t *n_out);

/* Queue of instance `id`, head first: sequence number, work and remaining
 * work (us) of each entry; *n_out = queue length.  Synchronous. */
DM_API dm_status dm_export_queue(dm_handle *h, uint32_t id, uint64_t *seq_host, uint64_t *work_host,
                          uint64_t *remaining_host, uint64_t cap, uint64_t *n_out);

/* Ring f (0-based: 0 or 1, or below dm_config.candidates on a handle made
 * for more candidates) as sorted (position, owner) arrays; *n_out = its
 * length.  Synchronous. */
DM_API dm_status dm_export_ring(dm_handle *h, int f, uint64_t *vpos_host, uint32_t *owner_host,
                         uint32_t cap, uint32_t *n_out);

/* Value of the global commit clock (number of block touches so far). */
DM_API dm_status dm_get_clock(dm_handle *h, uint64_t *clock_host);

/* Housekeeping of the per-instance cache indices since dm_create: how many
 * times an instance's key index was rebuilt (it would have passed half full,
 * counting the slots evicted keys keep) and how many times an instance's
 * recency log was compacted (it would have overflowed).  The paper has no
 * counterpart (its per-instance metadata store is opaque); neither changes
 * any routing result.  For tests and monitoring; read-only, synchronous,
 * works after a sticky error. */
DM_API dm_status dm_get_maint_counts(dm_handle *h, uint64_t *rebuilds_host, uint64_t *compactions_host);

/* Serving metrics kept on the device since dm_create or the last reset
 * (Sec. 2.2: load-balance CV; Sec. 4.1: cache hit rate, SLO attainment,
 * TTFT percentiles).  The time model is the scheduler's own: each queue
 * runs its work at one microsecond per microsecond from the batch times
 * on, so a request completes when the work ahead of it and its own is
 * done, and its TTFT is that moment minus its batch time (kept across
 * migrations).  Requests still queued are not counted as completed. */
#define DM_HIST_BUCKETS 976u   /* TTFT histogram: 0..15 exact, then 16 per power of two */
typedef struct {
    uint64_t requests;        /* routed requests */
    uint64_t prompt_tokens;   /* sum of their lengths */
    uint64_t hit_tokens;      /* sum of the cached-prefix tokens on the chosen instance at routing */
    uint64_t switched;        /* requests routed with switched = 1 */
    uint64_t est_slo_met;     /* requests whose estimated TTFT on the chosen instance
                                 (its load including the request) was <= SLO when routed */
    uint64_t completed;       /* requests whose prefill completed in a drain */
    uint64_t ttft_sum_us;     /* sum of their TTFTs */
    uint64_t ttft_max_us;
    uint64_t slo_met;         /* completed with TTFT <= SLO */
    uint64_t ttft_p50_us;     /* the lower edge of the histogram bucket holding the */
    uint64_t ttft_p90_us;     /* ceil(p * completed)-th smallest TTFT (0 if none); the */
    uint64_t ttft_p99_us;     /* bucket is at most 1/16 of its lower edge wide */
    uint64_t cv_samples;      /* batches with at least one request */
    double cv_sum;            /* sum over those batches of the CV of the live instances' W
                                 after the batch's choices: sqrt(n*S2 - S1^2) / S1 with
                                 S1 = sum W_i, S2 = sum W_i^2 (0 if S1 = 0) */
    double cv_last;           /* the last sample */
} dm_metrics;

/* Copy the metrics into *out_host and, if hist_host is not NULL, the first
 * min(hist_cap, DM_HIST_BUCKETS) TTFT histogram counts; bucket k holds
 * values v with v = k for k < 16, else e = floor(log2 v), k = 16 + 16(e-4) +
 * ((v >> (e-4)) & 15).  reset = 1 then clears them.  Synchronous; works
 * after a sticky error. */
DM_API dm_status dm_get_metrics(dm_handle *h, dm_metrics *out_host, uint64_t *hist_host, uint32_t hist_cap,
                                int reset);

/* Hash prefix length (blocks) each request of the last routed batch was
 * mapped with: min(K_route, n_blk), or the adaptive length.  Copies n
 * (<= that batch's size) values to out_dev (device).  Asynchronous. */
DM_API dm_status dm_get_route_blocks(dm_handle *h, uint32_t *out_dev, uint32_t n);

/* Expanded nodes of the adaptive prefix hotness tree (their keys, in
 * unspecified order); *n_out = their number (entries beyond cap are not
 * written).  0 nodes when the length is fixed.  Synchronous. */
DM_API dm_status dm_export_prefix_tree(dm_handle *h, uint64_t *keys_host, uint64_t cap, uint64_t *n_out);

/* The power-of-d-choices experiment behind DualMap's two candidates (App.
 * A.8): `trials` independent trials of m_balls balls into n_bins bins, each
 * ball placed in the least loaded of d uniformly random bins (ties to the
 * earlier choice); max_load_dev (device, `trials` entries) receives each
 * trial's maximum bin load (the deviation is that minus m/n).  Ball t's
 * choice k in trial s is floor(x * n_bins / 2^64) for x the (c+1)-th output
 * of SplitMix64(seed), c = (s * m_balls + t) * d + k.  No handle; work is
 * enqueued on `stream` (a cudaStream_t, NULL = legacy default stream).
 * 1 <= n_bins <= 256, 1 <= d <= 64, m_balls < 2^32; DM_ERR_INVALID_ARG
 * otherwise, DM_ERR_CUDA if the launch fails. */
DM_API dm_status dm_potc_max_loads(uint32_t n_bins, uint64_t m_balls, uint32_t d, uint32_t trials, uint64_t seed,
                                   uint32_t *max_load_dev, void *stream);

/* Testing only (no paper counterpart): after this call the library's
 * (n + 1)-th device allocation, counted over every handle of the process,
 * fails as if the device were out of memory (without calling the CUDA
 * allocator), so a test can check that dm_create, dm_add_instance and the
 * host-buffer entry points return DM_ERR_OOM and leave no handle state
 * behind.  n < 0 turns the failure off.  Not thread-safe against concurrent
 * allocating calls. */
DM_API void dm_test_fail_alloc(int64_t n);

/* Synchronise the stream and return the sticky error (DM_OK if none). */
DM_API dm_status dm_last_error(dm_handle *h);

/* CUDA-event timing of the stages of every subsequent call: on = 0 none,
 * 1 every stage, or DM_PROFILE_ONLY | (1 << DM_STAGE_x) | ... only the stages
 * named.  Events between kernels cost a little time of their own; any other
 * value returns DM_ERR_INVALID_ARG. */
#define DM_PROFILE_ONLY 0x100
DM_API dm_status dm_set_profiling(dm_handle *h, int on);

/* Synchronise, then return the summed milliseconds and call counts of each
 * stage since the last reset (arrays of DM_STAGE_COUNT); reset = 1 clears. */
DM_API dm_status dm_get_stage_times(dm_handle *h, double *ms_host, uint64_t *calls_host, int reset);

/* Human-readable name of a status code. */
DM_API const char *dm_status_string(dm_status s);

#ifdef __cplusplus
}
#endif

#endif /* DUALMAP_H */
