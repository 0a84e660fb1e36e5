// dm_internal.cuh -- device state layout and device helpers shared by the
// kernels of the DualMap routing library (sm_103a).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "../../include/dualmap.h"

namespace dm {

constexpr int kWarp = 32;
constexpr uint32_t kSegBlocks = 64;        // blocks hashed by one warp task
constexpr uint32_t kMaxInstances = 8192;
constexpr uint32_t kMaxRouteBlocks = 256;
constexpr uint32_t kTomb = 0xFFFFFFFFu;    // QEntry::moved of an entry migrated away
constexpr int kMaxLevels = 8;
constexpr uint32_t kEvChunk = 1024;      // log records per eviction / compaction chunk
constexpr uint32_t kRbChunk = 4096;      // index slots per rebuild chunk
constexpr uint64_t kSpinLimit = 1ull << 26; // bound of every data-dependent device loop
constexpr uint32_t kGroup = 8;           // consecutive blocks of a prompt homed in one 128-byte index line
constexpr uint32_t kMaxD = 8;            // rings (hash functions) of the d-candidate routing path
// Head segments per request in the routing kernel's hashing order (the
// routing prefix and the usual cached run: 24 x 64 blocks = 24,576 tokens at
// B = 16; at most 32, the carries of a head are one warp scan).
constexpr uint32_t kHeadSegs = 24;

// One queued request (56 bytes).
struct QEntry {
    uint64_t seq, work, remaining;
    uint32_t L, c1, c2, h1, h2;
    uint32_t moved;   // 0, or the rebalance call that moved it here, or kTomb
    uint64_t arrival; // batch time the request arrived with
    uint64_t koff;    // DM_REBALANCE_FRESH_HITS: ring position of its first block key on this instance
};

// Serving metrics (dm_metrics before the percentiles), updated by the
// choice kernels and the drain.  A choice kernel leaves its batch's load
// sums (S1 = sum W, S2 = sum W^2 over the live instances, n of them; exact
// 128-bit integers) pending; the next setup kernel, or dm_get_metrics,
// turns them into the batch's CV sample, so the floating-point steps stay
// off the choice kernel's tail.
constexpr uint32_t kHistBuckets = DM_HIST_BUCKETS;
struct DevMetrics {
    unsigned long long requests, prompt_tokens, hit_tokens, switched, est_slo_met;
    unsigned long long completed, ttft_sum, ttft_max, slo_met, cv_samples;
    double cv_sum, cv_last;
    unsigned long long pend, pend_n, pend_s1[2], pend_s2[2];   // [lo, hi]
    unsigned long long hist[kHistBuckets];
};

// Population CV of Sec. 2.2 from the exact sums: sqrt(n*S2 - S1^2) / S1
// (0 when S1 = 0); each 128-bit integer becomes double(hi) * 2^64 +
// double(lo), every step rounded to nearest.
__host__ __device__ inline double u128_as_double(unsigned __int128 x) {
#ifdef __CUDA_ARCH__
    return __dadd_rn(__dmul_rn(__ull2double_rn((uint64_t)(x >> 64)), 18446744073709551616.0),
                     __ull2double_rn((uint64_t)x));
#else
    const double hi = (double)(uint64_t)(x >> 64) * 18446744073709551616.0;   // exact
    return hi + (double)(uint64_t)x;
#endif
}

__host__ __device__ inline double load_cv(uint64_t n, unsigned __int128 S1, unsigned __int128 S2) {
    if (S1 == 0) return 0.0;
#ifdef __CUDA_ARCH__
    return __ddiv_rn(__dsqrt_rn(u128_as_double((unsigned __int128)n * S2 - S1 * S1)), u128_as_double(S1));
#else
    return __builtin_sqrt(u128_as_double((unsigned __int128)n * S2 - S1 * S1)) / u128_as_double(S1);
#endif
}

// Fold a pending CV sample into the running sum.  One thread.
__host__ __device__ inline void fold_cv(DevMetrics *m) {
    if (!m->pend) return;
    const unsigned __int128 S1 = ((unsigned __int128)m->pend_s1[1] << 64) | m->pend_s1[0];
    const unsigned __int128 S2 = ((unsigned __int128)m->pend_s2[1] << 64) | m->pend_s2[0];
    const double cv = load_cv(m->pend_n, S1, S2);
#ifdef __CUDA_ARCH__
    m->cv_sum = __dadd_rn(m->cv_sum, cv);
#else
    m->cv_sum = m->cv_sum + cv;
#endif
    m->cv_last = cv;
    m->cv_samples += 1;
    m->pend = 0;
}

// One index slot (16 bytes): a block key and 1 + the position of its latest
// record in the instance's recency log; key 0 marks an empty slot.  A key is
// resident while that position is at or after the log front.
//
// Placement: the index is cut into buckets of kGroup slots (one 128-byte
// line).  Block b of a prompt (b counted from the prompt's start) prefers
// slot (b & 7) of bucket A & mask & ~7, A being the key of block b & ~7 of
// the same prompt (its group anchor), so the 8 blocks of a group share one
// line: one random DRAM access instead of 8 (random single-slot atomics
// saturate far below line-local ones).  A key fixes its whole prefix and so
// its anchor: every key has one home.  Probe order of a key: the slots of its
// home bucket cyclically from its preferred one; then those of a second
// bucket derived from the home bucket's index (a group displaced from a full
// home bucket moves there together; a hashed bucket is far likelier to be
// empty than the adjacent one, which earlier displaced groups fill); then
// the buckets from one chosen by the key's own hash onwards, each likewise.
// (Prompts that share a prefix but diverge inside a group share that group's
// anchor: past the first two buckets the key hash spreads their overflow
// instead of piling it up.)
// Inserts take the first slot of that order that is empty, and slots never
// empty again (until the index is rebuilt into the other buffer), so a
// lookup ends at the first bucket with an empty slot.
struct __align__(16) Slot {
    uint64_t key, pos1;
};

// One recency-log record (16 bytes): the block key and the global clock
// stamp of the touch.  Records of an instance are in stamp order.
struct Rec {
    uint64_t key, stamp;
};

// A touch that the commit's first atomics did not settle (32 bytes): the
// preferred slot of bucket `bucket` of the key's probe order (0: the home
// bucket) holds the key with an older position (found = 1, x = the position
// value seen last) or another key (found = 0).  The touch kernel finishes it
// from there at the end of its 32 segments.
struct Deferred {
    uint64_t key, p, x;     // p: log position of the touch's record
    uint32_t home;
    uint16_t found, bucket;
};

// One node count of the adaptive prefix tree's current window (16 bytes):
// key 0 marks an empty slot.
struct AdCount {
    uint64_t key;
    uint32_t count, depth;   // requests that reached the node; its length in blocks
};

// Values one warp of the routing kernel publishes for the others, without
// fences: every record ends with chk, the xor of its other words and the
// batch's epoch mask E (a different value per routing call), so a reader
// that sees chk match knows every word is this batch's (a torn or stale
// read fails the check except with probability about 2^-64) and retries.
// A head segment's record (48 bytes): its f1 total t1, its f2 partial t2,
// the local f1 prefix value of its first block pf and of block K-1 when that
// block lies in it (pk), and px, the xor of all its blocks' local f1 prefix
// values as stored in plocal (a reader of those values checks them
// against it the same way).
struct __align__(16) SegPub {
    uint64_t t1, t2, pf, pk, px, chk;
};
// Per-batch values produced on the device.
struct BatchInfo {
    uint64_t total_blocks;
    uint32_t total_segs;
    uint32_t n;
    uint32_t head_segs;     // routing: head segments past the routing columns (the second part)
    uint32_t col_tasks;     // routing: n x the routing columns (the first part)
    uint32_t tasks;         // routing: tasks of the routing kernel (all three parts)
    uint32_t pad0;
    uint64_t clock_base;    // commit clock before this batch's touches
    uint32_t final_dirty;   // a rebalance moved a request of this batch
    uint32_t mc_chunks;     // log-compaction chunks of this commit
    uint32_t mr_chunks;     // index-rebuild chunks of this commit
    uint32_t both_over;     // a request of this batch estimated TTFT > SLO on both candidates
    uint32_t fix_n;         // routing: entries of the last CTA's list
    uint32_t cta_done;      // routing: CTAs of the routing kernel that finished
    uint32_t mt_done_a;     // commit: CTAs of k_maint_a that finished
    uint32_t mt_done_c;     // commit: CTAs of k_maint_c that finished
    uint32_t rb_rr_next;    // commit: rotation start of the rebuild order after this commit
};

struct Ring {
    uint64_t *vpos;       // sorted positions, R entries
    uint32_t *owner;      // owner id per entry
    uint32_t *vidx;       // virtual-node index per entry (tie order)
    uint64_t *tree;       // 32-ary search levels >= 1, concatenated
};

struct DevState {
    // configuration
    uint32_t B, Kroute, V, M;
    uint64_t C, slo;
    uint32_t cost, hot_num, hot_den, max_batch;
    uint32_t rule;                  // dm_choice_rule
    uint32_t rb_flags;              // DM_REBALANCE_*
    // adaptive prefix length (ad_step = 0: every request hashes min(Kroute, n_blk) blocks)
    uint32_t Kf2;                   // the f2 digests are hashed over blocks < min(Kf2, n_blk)
    uint32_t ad_step, ad_max;
    uint64_t *ad_set;               // expanded nodes: open addressing on the key, 0 = empty
    uint64_t ad_set_mask;
    AdCount *ad_cnt;                // node counts of the current window
    uint64_t ad_cnt_mask;
    uint64_t max_blocks, max_segs, T, S, logcap;
    uint64_t loop_limit;            // 0, or the test cap of the index's bucket walks and touch retries
    uint64_t rb_thr;                // an index is rebuilt when its taken slots would pass this
    uint32_t Q;
    // key material
    uint32_t K1[64], K2[64];
    uint64_t G1, G2, Sc, Sr1, Sr2, Sv1, Sv2;
    // functions 3..kMaxD of the d-candidate path: salts and seeds (index f - 2
    // for 0-based f >= 2), NH keys in device memory (64 words per function)
    uint64_t Gx[kMaxD - 2], Srx[kMaxD - 2], Svx[kMaxD - 2];
    const uint32_t *Kx;
    uint32_t nrings;                // rings kept: 2, or the d-candidate path's d when larger
    uint32_t nd;                    // candidates of the d-candidate path (0: DualMap's two)
    uint32_t *rd_cand, *rd_hit;     // d-candidate path: per request, nd candidates and their hit tokens
    // rings (all have R entries)
    Ring ring[kMaxD];
    uint32_t R, nlev;
    uint64_t lev_off[kMaxLevels];   // offset of level k (k >= 1) inside tree
    uint64_t lev_n[kMaxLevels];     // entries in level k (lev_n[0] = R)
    uint8_t *inst_state;            // 0 absent, 1 live, 2 draining
    uint32_t *next_live;
    // per instance
    uint64_t *W;
    uint32_t *q_head, *q_tail;
    QEntry *q;                      // M x Q
    Slot **table;                   // per id: S slots (null until first add)
    Rec **logbuf;                   // per id: logcap records
    uint8_t **stale;                // per id: logcap flags, 1 = record superseded by a later touch
    uint32_t **loghome;             // per id: logcap index home slots, one per record
    Slot **table_alt;               // per id: its rebuild target during a commit that rebuilds it, else null
    Slot **pool;                    // spare index buffers shared by all ids (pool_n of them)
    uint32_t pool_n;
    uint32_t *rb_slot;              // per id: the pool entry its rebuild took this commit
    uint32_t *rb_rr;                // round-robin start of the rebuild order (1 entry)
    Rec **logbuf_alt;               // per id: second log buffer (compaction target)
    uint8_t **stale_alt;
    uint32_t **loghome_alt;
    uint64_t *log_front, *log_tail, *live, *used;
    // maintenance plan: per id flags / new log tail, chunk offsets and counts
    uint32_t *mt_flags;
    uint64_t *mt_newtail;
    uint32_t *mc_chunk_off, *mr_chunk_off;   // M + 1 entries each
    uint32_t *mc_chunk_live;
    uint64_t mc_cap;                         // compaction chunks that fit
    // batch scratch
    uint32_t *r_L, *r_nblk, *r_segoff;
    uint64_t *r_tokoff, *r_blkoff;
    uint32_t *seg_req;
    // routing order of the hashing tasks: the routing columns (segment j < Ccols
    // of every request), then the rest of each request's head (segments
    // below H), then the rest; per request the exclusive offsets of the last
    // two parts
    uint32_t H, Ccols;              // head segments, routing columns (segments holding any routing prefix)
    uint32_t *r_hoff, *r_toff;
    // routing kernel's exchange between warps (see dm_hash.cu): what each
    // head segment publishes, each request's first miss on each candidate
    // (0xFFFFFFFF: the whole prompt is resident), and the route tasks left
    // to the kernel's last CTA
    SegPub *seg_pub;
    uint32_t *r_m1, *r_m2;
    // DM_REBALANCE_FRESH_HITS (KQ = 0 otherwise): per instance a ring of KQ
    // block keys of its queued requests (instance i's at kring + i KQ), with
    // monotonic head and tail positions; per request of the pending batch
    // the ring position of its keys on its final instance
    uint64_t KQ;
    uint64_t *kring, *kr_head, *kr_tail, *r_koff;
    uint32_t *rb_hq;                // rebalance scratch: a candidate's hit on its other candidate, per queue slot
    uint64_t *fix_list;             // queue entries of route tasks (request, tries)
    uint64_t *seg_total, *seg_carry, *plocal;
    uint64_t *p2local;              // adaptive only: per block < Kf2, in-segment prefix of its f2 digests
    uint32_t *r_K;                  // per request: the hash prefix length it was routed with
    uint64_t *seg_total2;           // per segment: f2 digest sum over its blocks < K
    Deferred *defer;                // kSegBlocks per segment: touches the commit's first atomics left open
    uint32_t *r_c1, *r_c2, *r_final;
    uint64_t *r_touchoff;           // per request: offset among its instance's records of the batch
    uint64_t *log_adv;              // per id: log records the pending batch appends
    uint64_t *log_base;             // per id: log tail when the commit starts
    BatchInfo *info;
    uint64_t *clock;
    uint64_t *maint_count;          // index rebuilds and log compactions so far (2 counters)
    uint32_t *err;
    uint64_t *seq_next;
    DevMetrics *metrics;
    uint32_t *h_all;                // max_batch x M hit tokens (cluster-wide rules only)
    // rebalance scratch
    uint64_t *rb_key;               // sort keys (benefit, biased) per candidate
    uint64_t *rb_seq;
    uint64_t *rb_ttft;
    uint32_t *rb_pos;               // queue position of the candidate
    uint32_t rb_cap;                // candidates that fit (power of two)
};

// ---------------------------------------------------------------------------
// Programmatic dependent launch.  The kernels of the routing and commit path
// begin with pdl_enter(): the stream's next kernel may be launched as soon
// as all of this kernel's CTAs are running (its CTAs then wait at their own
// pdl_enter), and nothing here touches memory before the previous kernel
// has completed with its writes visible.  So the order of the stream is
// kept and only the launch latency between kernels is hidden.
__device__ __forceinline__ void pdl_enter() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

// Return the first failing launch of a launcher function.
#define DM_TRY(x)                            \
    do {                                     \
        const cudaError_t dm_e_ = (x);       \
        if (dm_e_ != cudaSuccess) return dm_e_; \
    } while (0)

// Launch a kernel that begins with pdl_enter() with programmatic stream
// serialization.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), unsigned grid, unsigned block, size_t smem, cudaStream_t st,
                              Args... args) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(block);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at{};
    at.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at.val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = &at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// ---------------------------------------------------------------------------
// Published mixers.
// MurmurHash3 64-bit finaliser (Appleby, public domain).
__device__ __host__ __forceinline__ uint64_t fmix64(uint64_t k) {
    k ^= k >> 33;
    k *= 0xff51afd7ed558ccdULL;
    k ^= k >> 33;
    k *= 0xc4ceb9fe1a85ec53ULL;
    k ^= k >> 33;
    return k;
}

// One SplitMix64 output step from state x (Steele, Lea & Flood 2014).
__device__ __host__ __forceinline__ uint64_t splitmix_step(uint64_t x) {
    uint64_t z = x + 0x9E3779B97F4A7C15ULL;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

// Cache key of a block from its chained prefix value (0 is the empty slot).
__device__ __forceinline__ uint64_t cache_key(uint64_t P, uint64_t Sc) {
    uint64_t k = fmix64(P ^ Sc);
    return k ? k : 1ull;
}

// Virtual-node position of (id, v) on a ring with seed Sv.
__device__ __host__ __forceinline__ uint64_t vnode_pos(uint64_t Sv, uint32_t id, uint32_t v) {
    return fmix64(splitmix_step((uint64_t(id) << 32) | v) ^ Sv);
}

// First error wins; kernels of a call stop at entry once it is set.
__device__ __forceinline__ void set_err(uint32_t *err, uint32_t code) {
    atomicCAS(err, 0u, code);
}

__device__ __forceinline__ bool has_err(const uint32_t *err) {
    return *(volatile const uint32_t *)err != 0u;
}

// Debug builds (-DDM_DEBUG, libdualmap_debug.so): DM_CHECK records
// DM_ERR_BOUNDS when an index invariant that the release build relies on
// does not hold, and DM_CLAMP also keeps the access inside its buffer.
// Nothing traps: the call ends with the sticky status.  Release builds
// compile both to nothing (DM_CLAMP to the index itself).
#ifdef DM_DEBUG
#define DM_CHECK(cond, err)                                     \
    do {                                                        \
        if (!(cond)) ::dm::set_err((err), DM_ERR_BOUNDS);       \
    } while (0)
__device__ __forceinline__ uint64_t dm_clamp(uint64_t i, uint64_t n, uint32_t *err) {
    if (i < n) return i;
    set_err(err, DM_ERR_BOUNDS);
    return n ? n - 1 : 0;
}
#define DM_CLAMP(i, n, err) ::dm::dm_clamp((i), (n), (err))
#else
#define DM_CHECK(cond, err) \
    do {                    \
    } while (0)
#define DM_CLAMP(i, n, err) (i)
#endif

__device__ __forceinline__ uint64_t shfl_u64(uint64_t v, int src) {
    return __shfl_sync(0xffffffffu, v, src);
}

__device__ __forceinline__ uint64_t shfl_xor_u64(uint64_t v, int m) {
    return __shfl_xor_sync(0xffffffffu, v, m);
}

__device__ __forceinline__ uint64_t shfl_up_u64(uint64_t v, int d) {
    return __shfl_up_sync(0xffffffffu, v, d);
}

// Inclusive warp scan of uint64 values (mod 2^64).
__device__ __forceinline__ uint64_t warp_incl_scan(uint64_t v, int lane) {
#pragma unroll
    for (int d = 1; d < kWarp; d <<= 1) {
        uint64_t u = shfl_up_u64(v, d);
        if (lane >= d) v += u;
    }
    return v;
}

// 16-byte slot load that bypasses L1 (probes are random; L2 is the cache).
__device__ __forceinline__ Slot load_slot(const Slot *p) {
    Slot s;
    asm volatile("ld.global.cg.v2.u64 {%0, %1}, [%2];"
                 : "=l"(s.key), "=l"(s.pos1) : "l"(__cvta_generic_to_global(p)));
    return s;
}

// Home slot of block b given its group anchor's key.
__device__ __forceinline__ uint64_t group_home(uint64_t anchor, uint64_t b, uint64_t mask) {
    return (anchor & mask & ~uint64_t(kGroup - 1)) | (b & (kGroup - 1));
}

// Bucket j >= 1 of the probe order of key (bucket 0 is its home bucket R0):
// j = 1 the bucket derived from R0 (the one after R0 should they coincide);
// j >= 2 the bucket chosen by the key's hash, then those after it.
constexpr uint64_t kLinearBuckets = 2;
__device__ __forceinline__ uint64_t probe_bucket(uint64_t j, uint64_t R0, uint64_t key, uint64_t mask) {
    if (j == 1) {
        const uint64_t R1 = fmix64(R0 ^ 0x5bd1e995a4c3b2e1ull) & mask & ~uint64_t(kGroup - 1);
        return R1 == R0 ? (R0 + kGroup) & mask : R1;
    }
    return ((fmix64(key) & mask & ~uint64_t(kGroup - 1)) + (j - kLinearBuckets) * kGroup) & mask;
}

// Key of the group anchor of the block held by this lane, when consecutive
// lanes hold consecutive blocks and lane 0 holds a block of group boundary.
// Whole warp.
__device__ __forceinline__ uint64_t group_anchor(uint64_t key, int lane) {
    return __shfl_sync(0xffffffffu, key, lane & ~int(kGroup - 1));
}

// Look key up in one instance's index from its home slot: its slot index
// and contents, or kNoSlot.  The home slot is read first (it usually
// settles the lookup); otherwise whole buckets are read at once.
constexpr uint64_t kNoSlot = ~0ull;
__device__ __forceinline__ uint64_t table_find(const Slot *t, uint64_t mask, uint64_t key, uint64_t home,
                                               uint32_t *err, Slot *found, uint64_t loop_limit = 0) {
    const Slot h = load_slot(t + home);
    if (h.key == key) { *found = h; return home; }
    if (h.key == 0) return kNoSlot;
    const uint64_t R0 = home & ~uint64_t(kGroup - 1);
    uint64_t R = R0;
    uint64_t walk = (mask >> 3) + kLinearBuckets + 1;
    if (loop_limit && loop_limit < walk) walk = loop_limit;
    for (uint64_t nbk = 1; nbk <= walk; ++nbk) {
        Slot sn[kGroup];
#pragma unroll
        for (int j = 0; j < (int)kGroup; ++j) sn[j] = load_slot(t + R + j);
        bool empty = false;
        uint64_t hit = kNoSlot;
        Slot hs{0, 0};
#pragma unroll
        for (int j = 0; j < (int)kGroup; ++j) {
            if (sn[j].key == key) { hit = R + j; hs = sn[j]; }
            empty |= sn[j].key == 0;
        }
        if (hit != kNoSlot) { *found = hs; return hit; }
        if (empty) return kNoSlot;
        R = probe_bucket(nbk, R0, key, mask);
    }
    set_err(err, DM_ERR_TIMEOUT);
    return kNoSlot;
}

// 1 + log position of key's latest record (0 if the key has no slot).
__device__ __forceinline__ uint64_t table_pos1(const Slot *t, uint64_t mask, uint64_t key, uint64_t home,
                                               uint32_t *err, uint64_t loop_limit = 0) {
    Slot s;
    return table_find(t, mask, key, home, err, &s, loop_limit) == kNoSlot ? 0 : s.pos1;
}

// Carries of one request's segments (exclusive prefix of the segment
// totals written by the hashing kernel), stored in seg_carry.  Whole warp.
__device__ __forceinline__ void request_carries(const DevState &d, uint32_t r, int lane) {
    const uint32_t s0 = d.r_segoff[r];
    const uint32_t ns = (d.r_nblk[r] + kSegBlocks - 1) / kSegBlocks;
    uint64_t carry = 0;
    for (uint32_t b = 0; b < ns; b += 32) {
        const uint32_t s = b + lane;
        const uint64_t t = s < ns ? d.seg_total[s0 + s] : 0;
        const uint64_t inc = warp_incl_scan(t, lane);
        if (s < ns) d.seg_carry[s0 + s] = carry + inc - t;
        carry += shfl_u64(inc, 31);
    }
}

// Cached-prefix tokens on a candidate: B x the leading run of resident
// blocks, from the first missing block found by the routing kernel
// (0xFFFFFFFF: no block of the prompt missed).
__device__ __forceinline__ uint32_t hit_tokens(uint32_t first_miss, uint32_t nblk, uint32_t B) {
    return (first_miss < nblk ? first_miss : nblk) * B;
}

// After the routing kernel, a warp per request, for a kernel whose CTAs
// cta = 0..nctas-1 take this role: the carries of every segment (the
// commit needs them) and the request's route outputs.
__device__ __forceinline__ void carries_role(const DevState &d, const dm_route_out &o, uint32_t n, uint32_t cta,
                                             uint32_t nctas) {
    const int lane = threadIdx.x & 31;
    const uint32_t wpc = blockDim.x >> 5;
    for (uint32_t r = cta * wpc + (threadIdx.x >> 5); r < n; r += nctas * wpc) {
        request_carries(d, r, lane);
        if (lane == 0) {
            const uint32_t nblk = d.r_nblk[r];
            o.cand1[r] = d.r_c1[r];
            o.cand2[r] = d.r_c2[r];
            o.hit1[r] = hit_tokens(d.r_m1[r], nblk, d.B);
            o.hit2[r] = hit_tokens(d.r_m2[r], nblk, d.B);
        }
    }
}

// The two ring positions of request r (after request_carries): P^1_{K-1}
// from its local prefix value plus carry, P^2_{K-1} as the sum of the f2
// segment partials (f2 only runs over blocks < K).  Whole warp; all lanes
// return the same values.
__device__ __forceinline__ void route_positions(const DevState &d, uint32_t r, int lane, uint64_t &pos1,
                                                uint64_t &pos2) {
    const uint32_t nblk = d.r_nblk[r], s0 = d.r_segoff[r];
    const uint32_t K = min(d.Kroute, nblk);
    const uint32_t last = (K - 1) / kSegBlocks;   // segments holding blocks < K: 0..last
    const uint64_t P1 = d.plocal[d.r_blkoff[r] + K - 1] + d.seg_carry[s0 + last];
    uint64_t p2 = 0;
    for (uint32_t j = lane; j <= last; j += 32) p2 += d.seg_total2[s0 + j];
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) p2 += shfl_xor_u64(p2, o);
    pos1 = fmix64(P1 ^ d.Sr1);
    pos2 = fmix64(p2 ^ d.Sr2);
}

// ---------------------------------------------------------------------------
// Adaptive prefix tree tables (open addressing, linear probing, bounded).

__device__ __forceinline__ uint64_t ad_slot(uint64_t key, uint64_t mask) {
    return fmix64(key ^ 0x2545F4914F6CDD1Dull) & mask;
}

__device__ __forceinline__ bool ad_set_contains(const uint64_t *set, uint64_t mask, uint64_t key, uint32_t *err) {
    uint64_t x = ad_slot(key, mask);
    for (uint64_t i = 0; i <= mask; ++i, x = (x + 1) & mask) {
        const uint64_t k = set[x];
        if (k == key) return true;
        if (k == 0) return false;
    }
    set_err(err, DM_ERR_CAPACITY);
    return false;
}

__device__ __forceinline__ void ad_set_insert(uint64_t *set, uint64_t mask, uint64_t key, uint32_t *err) {
    uint64_t x = ad_slot(key, mask);
    for (uint64_t i = 0; i <= mask; ++i, x = (x + 1) & mask) {
        const unsigned long long k = atomicCAS(reinterpret_cast<unsigned long long *>(set + x), 0ull,
                                               (unsigned long long)key);
        if (k == 0 || k == key) return;
    }
    set_err(err, DM_ERR_CAPACITY);
}

// One more request reached node `key` (length `depth` blocks).
__device__ __forceinline__ void ad_count_add(AdCount *cnt, uint64_t mask, uint64_t key, uint32_t depth,
                                             uint32_t *err) {
    uint64_t x = ad_slot(key, mask);
    for (uint64_t i = 0; i <= mask; ++i, x = (x + 1) & mask) {
        const unsigned long long k = atomicCAS(reinterpret_cast<unsigned long long *>(&cnt[x].key), 0ull,
                                               (unsigned long long)key);
        if (k == 0 || k == key) {
            if (k == 0) cnt[x].depth = depth;
            atomicAdd(&cnt[x].count, 1u);
            return;
        }
    }
    set_err(err, DM_ERR_CAPACITY);
}

__device__ __forceinline__ uint32_t ad_count_get(const AdCount *cnt, uint64_t mask, uint64_t key, uint32_t *err) {
    uint64_t x = ad_slot(key, mask);
    for (uint64_t i = 0; i <= mask; ++i, x = (x + 1) & mask) {
        const uint64_t k = cnt[x].key;
        if (k == key) return cnt[x].count;
        if (k == 0) return 0;
    }
    set_err(err, DM_ERR_CAPACITY);
    return 0;
}

// ---------------------------------------------------------------------------
// Metrics helpers.

// TTFT histogram bucket: v < 16 exact; else e = floor(log2 v) and the four
// bits below the top one select one of 16 buckets of [2^e, 2^(e+1)).
__device__ __forceinline__ uint32_t hist_bucket(uint64_t v) {
    if (v < 16) return (uint32_t)v;
    const uint32_t e = 63 - __clzll((long long)v);
    return 16 + 16 * (e - 4) + (uint32_t)((v >> (e - 4)) & 15);
}

__device__ __forceinline__ uint64_t warp_sum_u64(uint64_t v) {
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) v += shfl_xor_u64(v, o);
    return v;
}

__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) v = max(v, shfl_xor_u64(v, o));
    return v;
}

// Completed requests of one warp step: lanes with fin set finished with
// TTFT ttft.  Whole warp.
__device__ __forceinline__ void record_completions(DevMetrics *m, bool fin, uint64_t ttft, uint64_t slo,
                                                   int lane) {
    const uint32_t fm = __ballot_sync(0xffffffffu, fin);
    if (!fm) return;
    if (fin) atomicAdd(&m->hist[hist_bucket(ttft)], 1ull);
    const uint64_t sum = warp_sum_u64(fin ? ttft : 0);
    const uint64_t mx = warp_max_u64(fin ? ttft : 0);
    const uint32_t met = __popc(__ballot_sync(0xffffffffu, fin && ttft <= slo));
    if (lane == 0) {
        atomicAdd(&m->completed, (unsigned long long)__popc(fm));
        atomicAdd(&m->ttft_sum, (unsigned long long)sum);
        atomicMax(&m->ttft_max, (unsigned long long)mx);
        if (met) atomicAdd(&m->slo_met, (unsigned long long)met);
    }
}

// Run `delta` us of prefill work off the head of instance i's queue (Sec.
// 3.2: an instance's load is its pending prefill work).  Whole warp.
__device__ __forceinline__ void drain_queue(const DevState &d, uint32_t i, uint64_t delta, uint64_t t0,
                                            int lane) {
    uint32_t head = d.q_head[i];
    const uint32_t tail = d.q_tail[i];
    if (head == tail) return;
    const QEntry *qb = d.q + uint64_t(i) * d.Q;
    uint64_t left = delta, used = 0;
    while (head != tail) {
        const uint32_t cnt = min(32u, tail - head);
        const uint32_t idx = (head + lane) & (d.Q - 1);
        const bool valid = (uint32_t)lane < cnt;
        const uint64_t rem = valid ? qb[idx].remaining : 0;
        const uint32_t moved = valid ? qb[idx].moved : 0;
        const uint64_t arrival = valid ? qb[idx].arrival : 0;
        const uint64_t inc = warp_incl_scan(rem, lane);
        const uint32_t done = __ballot_sync(0xffffffffu, valid && inc <= left);
        const uint32_t ndone = __popc(done);   // a prefix of the lanes
        // Entry `lane` completes `used + inc` us into the window that starts
        // at t0; migrated-away entries (no work left here) are not requests.
        const bool fin = ((done >> lane) & 1u) && moved != kTomb;
        record_completions(d.metrics, fin, fin ? t0 + used + inc - arrival : 0, d.slo, lane);
        if (ndone == cnt) {                    // whole chunk drained
            const uint64_t tot = shfl_u64(inc, 31);
            left -= tot;
            used += tot;
            head += cnt;
            continue;
        }
        const uint64_t before = ndone ? shfl_u64(inc, ndone - 1) : 0;
        if ((uint32_t)lane == ndone) {
            const uint64_t take = left - before;   // < rem of this entry
            d.q[uint64_t(i) * d.Q + idx].remaining = rem - take;
        }
        used += left;
        left = 0;
        head += ndone;
        break;
    }
    if (lane == 0) {
        d.q_head[i] = head;
        d.W[i] -= used;
        if (d.KQ) d.kr_head[i] = head != tail ? qb[head & (d.Q - 1)].koff : d.kr_tail[i];
    }
}

// The same two ring positions without the stored carries: the carry of the
// segment holding block K-1 is summed here from the (at most 4) segment
// totals before it, so the ring search need not wait for request_carries.
// Whole warp; all lanes return the same values.
__device__ __forceinline__ void route_positions_direct(const DevState &d, uint32_t r, int lane, uint64_t &pos1,
                                                       uint64_t &pos2) {
    const uint32_t nblk = d.r_nblk[r], s0 = d.r_segoff[r];
    const uint32_t K = min(d.Kroute, nblk);
    const uint32_t last = (K - 1) / kSegBlocks;   // <= 3 (K <= 256)
    uint64_t c = (uint32_t)lane < last ? d.seg_total[s0 + lane] : 0;
    uint64_t p2 = (uint32_t)lane <= last ? d.seg_total2[s0 + lane] : 0;
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
        c += shfl_xor_u64(c, o);
        p2 += shfl_xor_u64(p2, o);
    }
    const uint64_t P1 = d.plocal[d.r_blkoff[r] + K - 1] + c;
    pos1 = fmix64(P1 ^ d.Sr1);
    pos2 = fmix64(p2 ^ d.Sr2);
}

// ---------------------------------------------------------------------------
// Routing helpers (Sec. 3.2, Sec. 3.4, App. A.1.3, App. A.3.2).

__device__ __forceinline__ const uint64_t *level_ptr(const DevState &d, int f, int k) {
    return k == 0 ? d.ring[f].vpos : d.ring[f].tree + d.lev_off[k];
}

// Ring search.  Each ring is a sorted array of virtual-node positions plus a
// static 32-ary search tree (level k holds every 32^k-th position).  A warp
// compares one 256-byte row of 32 keys per level and ballots, so a ring of
// 262,144 nodes takes four coalesced L2 reads.  The successor of p is the
// first node with position >= p, wrapping to node 0.  Returns the level-0
// index of the successor of p1 on ring 0 and of p2 on ring 1; whole warp,
// the two searches interleaved for memory-level parallelism.
__device__ __forceinline__ void ring_search2(const DevState &d, uint64_t p1, uint64_t p2, int lane,
                                             uint32_t &lb1, uint32_t &lb2) {
    const int top = (int)d.nlev - 1;
    int64_t i1, i2;
    {
        const uint64_t nt = d.lev_n[top];
        const uint64_t v1 = (uint64_t)lane < nt ? level_ptr(d, 0, top)[lane] : ~0ull;
        const uint64_t v2 = (uint64_t)lane < nt ? level_ptr(d, 1, top)[lane] : ~0ull;
        i1 = (int64_t)__popc(__ballot_sync(0xffffffffu, v1 < p1)) - 1;
        i2 = (int64_t)__popc(__ballot_sync(0xffffffffu, v2 < p2)) - 1;
    }
    for (int k = top - 1; k >= 0; --k) {
        const uint64_t nk = d.lev_n[k];
        const uint64_t a1 = (uint64_t)(i1 < 0 ? 0 : i1) * 32 + lane;
        const uint64_t a2 = (uint64_t)(i2 < 0 ? 0 : i2) * 32 + lane;
        const uint64_t v1 = (i1 >= 0 && a1 < nk) ? level_ptr(d, 0, k)[a1] : ~0ull;
        const uint64_t v2 = (i2 >= 0 && a2 < nk) ? level_ptr(d, 1, k)[a2] : ~0ull;
        const int c1 = __popc(__ballot_sync(0xffffffffu, v1 < p1));
        const int c2 = __popc(__ballot_sync(0xffffffffu, v2 < p2));
        if (i1 >= 0) i1 = i1 * 32 + c1 - 1;
        if (i2 >= 0) i2 = i2 * 32 + c2 - 1;
    }
    lb1 = (uint32_t)(i1 + 1 == (int64_t)d.R ? 0 : i1 + 1);
    lb2 = (uint32_t)(i2 + 1 == (int64_t)d.R ? 0 : i2 + 1);
}

// Is key resident on an instance (log front `front`), given s0, the slot
// already read at its home?  The home slot settles most lookups.
__device__ __forceinline__ bool resident_at(const Slot *t, uint64_t mask, uint64_t key, uint64_t home,
                                            uint64_t front, const Slot &s0, uint32_t *err, uint64_t loop_limit = 0) {
    if (s0.key == key) return s0.pos1 > front;
    if (s0.key == 0) return false;
    return table_pos1(t, mask, key, home, err, loop_limit) > front;
}

// Adaptive hash-prefix length (Sec. 3.2): the walk from min(K_route, n_blk)
// blocks, one step deeper while the node (the key of the prefix's last
// block) is expanded.  Level j sits at depth min(d0 + j * step, cap), so
// lane j evaluates level j of each 32-level round at once: the request's
// length is the first level that cannot extend.  Every level passed and the
// final one count toward the window's hotness.  Then the two positions of
// that length.  c1, c2: lane s holds the carry (exclusive prefix of the
// segment totals) of segment s of the request under f1 and f2, for every
// segment below the cap (at most 32: ad_max <= 2048).  Whole warp.  The
// prefix values are read through L2 (they may have been written by other
// warps of the calling kernel).
__device__ __forceinline__ void adaptive_positions(const DevState &d, uint32_t r, uint32_t nblk, uint64_t bo,
                                                   int lane, uint64_t c1, uint64_t c2, uint64_t &pos1,
                                                   uint64_t &pos2, uint32_t &Kout) {
    const uint32_t d0 = min(d.Kroute, nblk), cap = min(d.ad_max, nblk);
    uint32_t K = d0;
    uint64_t P1K = 0;
    for (uint32_t j0 = 0;; j0 += 32) {
        const uint64_t want = uint64_t(d0) + uint64_t(j0 + lane) * d.ad_step;
        const uint32_t dj = want < cap ? (uint32_t)want : cap;
        const uint32_t b = dj - 1;
        const uint64_t P1 = __ldcg(d.plocal + bo + b) + shfl_u64(c1, b / kSegBlocks);
        const uint64_t key = cache_key(P1, d.Sc);
        const bool ext = dj < cap && ad_set_contains(d.ad_set, d.ad_set_mask, key, d.err);
        const uint32_t stop = __ballot_sync(0xffffffffu, !ext);
        const int last = stop ? __ffs(stop) - 1 : 31;   // levels of this round that count
        if (lane <= last) ad_count_add(d.ad_cnt, d.ad_cnt_mask, key, dj, d.err);
        if (stop) {
            K = __shfl_sync(0xffffffffu, dj, last);
            P1K = shfl_u64(P1, last);
            break;
        }
    }
    const uint64_t P2K = __ldcg(d.p2local + bo + K - 1) + shfl_u64(c2, (K - 1) / kSegBlocks);
    pos1 = fmix64(P1K ^ d.Sr1);
    pos2 = fmix64(P2K ^ d.Sr2);
    Kout = K;
}

// Streaming multiprocessors of the current device.
inline int sm_count() {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    return sms > 0 ? sms : 1;
}

// Grid of a grid-stride kernel: every SM filled to the kernel's occupancy.
template <typename K>
inline int full_grid(K kernel, int block) {
    int dev = 0, sms = 0, per = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, kernel, block, 0);
    return sms * (per > 0 ? per : 1);
}

// ---------------------------------------------------------------------------
// Host-side launchers (one translation unit each).
cudaError_t launch_setup(const DevState &d, const dm_batch &b, cudaStream_t st);
cudaError_t launch_hash(const DevState &d, const dm_batch &b, int grid, cudaStream_t st);
int hash_grid_size();
cudaError_t launch_setup_route(const DevState &d, const dm_batch &b, uint64_t delta, uint64_t t0,
                               cudaStream_t st);
cudaError_t launch_setup_plain_drain(const DevState &d, const dm_batch &b, uint64_t delta, uint64_t t0,
                                     cudaStream_t st);
cudaError_t launch_route_d(const DevState &d, const dm_batch &b, const dm_route_out_d &o, uint64_t seq0,
                           cudaStream_t st);
cudaError_t launch_shard_copy(const DevState &d, bool exp, uint32_t r0, uint32_t r1, uint8_t *buf, uint64_t cap,
                              uint64_t *bytes, cudaStream_t st);
cudaError_t launch_hash_probe(const DevState &d, const dm_batch &b, uint64_t E, uint32_t r0, uint32_t r1,
                              cudaStream_t st);
cudaError_t launch_carries(const DevState &d, const dm_route_out &o, uint32_t n, cudaStream_t st);
cudaError_t launch_adapt_update(const DevState &d, uint64_t *new_set, uint64_t n_live, uint64_t T, cudaStream_t st);
cudaError_t launch_choice(const DevState &d, const dm_route_out &o, uint32_t n, uint64_t seq0,
                          uint64_t t_batch, cudaStream_t st);
cudaError_t launch_commit(const DevState &d, uint32_t n, cudaStream_t st);
cudaError_t launch_rebalance(const DevState &d, uint32_t n, uint64_t seq0, uint32_t call,
                             dm_migration *out, uint32_t cap, uint32_t *n_out, cudaStream_t st);
cudaError_t launch_hash_keys(const DevState &d, uint32_t n, uint64_t *keys, uint64_t *key_off,
                             uint64_t *pos, cudaStream_t st);
cudaError_t launch_ring_lookup(const DevState &d, const uint64_t *pos, uint32_t n, uint32_t *o1,
                               uint32_t *o2, cudaStream_t st);
cudaError_t launch_ring_update(DevState &d, uint32_t id, bool add, uint64_t *scratch_pos, uint32_t *scratch_vidx,
                               uint64_t *const *new_vpos, uint32_t *const *new_owner, uint32_t *const *new_vidx,
                               cudaStream_t st);
cudaError_t launch_tree_build(const DevState &d, cudaStream_t st);
cudaError_t launch_next_live(const DevState &d, cudaStream_t st);
cudaError_t launch_set_state(const DevState &d, uint32_t id, uint8_t s, cudaStream_t st);

}  // namespace dm
