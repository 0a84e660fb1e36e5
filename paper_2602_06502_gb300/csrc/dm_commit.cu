// dm_commit.cu -- cache save with exact LRU eviction (App. A.3.2 "KV cache
// save"; each instance keeps a bounded index of cached prefix blocks).
//
// Sequential definition: in arrival order, each request of the batch touches
// its block keys on its final instance from block n_blk-1 down to 0, one
// global clock tick per touch, and an LRU of capacity C evicts on overflow.
// An LRU holds exactly the C distinct keys with the latest last touch, so all
// touches of a batch are applied at once and each instance then drops its
// oldest keys down to C.
//
// Layout per instance: a recency log of (key, stamp) records in stamp order,
// a stale flag per record (set when a later touch supersedes it), and an
// open-addressed index key -> 1 + position of the key's latest record.  A
// key is resident iff that record is at or after the log front, so evicting
// the k oldest keys is moving the front past the k-th non-stale record: no
// per-key write at all.  Evicted keys keep their index slots until the index
// passes its rebuild threshold, when it is rebuilt from the log's live records; a log
// about to overflow is compacted.  Both write into second buffers and swap.
#include <cooperative_groups.h>

#include "dm_internal.cuh"

namespace cg = cooperative_groups;

namespace dm {

constexpr int kMtThreads = 256;
constexpr uint32_t kPrepChunk = 1024;
constexpr uint32_t kFlagCompact = 1, kFlagRebuild = 2;
constexpr uint32_t kZeroChunk = 4096;   // slots or flag bytes cleared per chunk

// Raise the position word of a slot whose key is set (keys never change once
// set, and positions only grow): returns the value it had before.
__device__ __forceinline__ uint64_t pos_max(Slot *s, uint64_t p1) {
    return atomicMax(reinterpret_cast<unsigned long long *>(&s->pos1), (unsigned long long)p1);
}

// 16-byte compare-and-swap of a whole index slot; returns its previous
// contents.  Every claim of a slot by the touch kernel goes through this, so
// key and position are set together and never tear (whole-bucket reads are
// plain 16-byte loads used only to pick the next slot to try).
__device__ __forceinline__ Slot slot_cas(Slot *s, Slot expect, Slot desired) {
    Slot old;
    asm volatile(
        "{\n\t.reg .b128 c, v, r;\n\t"
        "mov.b128 c, {%2, %3};\n\t"
        "mov.b128 v, {%4, %5};\n\t"
        "atom.relaxed.gpu.global.cas.b128 r, [%6], c, v;\n\t"
        "mov.b128 {%0, %1}, r;\n\t}"
        : "=l"(old.key), "=l"(old.pos1)
        : "l"(expect.key), "l"(expect.pos1), "l"(desired.key), "l"(desired.pos1),
          "l"(__cvta_generic_to_global(s))
        : "memory");
    return old;
}

// Finish the touch of `key` at position value p1 (1 + log position), given
// `old`, the result of CAS({0,0} -> {key, p1}) at its home slot.  An empty
// slot was claimed by that CAS; a slot holding the key has its position
// raised to p1 unless a larger one is already there (a 64-bit atomic max on
// the position word: the slot's key never changes); a slot of another key moves on along the key's probe
// order, using a snapshot of the bucket to skip the slots other keys hold
// (slots never empty again, so only empty or matching ones are candidates).
// Every touch of a key follows the same order, so concurrent first touches
// meet at the same slot and one CAS wins.  Returns the position value the
// key had before (0 if claimed now).
__device__ __forceinline__ uint64_t touch_resolve(Slot *t, uint64_t mask, uint64_t key, uint64_t p1, uint64_t home,
                                                  Slot old, uint32_t *err, bool *claimed, uint32_t nbk0 = 0,
                                                  uint64_t loop_limit = 0) {
    // `old` was seen at the preferred slot of bucket nbk0 of the key's order
    const uint32_t o = (uint32_t)(home & (kGroup - 1));
    const uint64_t R0 = home & ~uint64_t(kGroup - 1);
    uint64_t nbk = nbk0;   // position of bucket R in the probe order
    uint64_t R = nbk0 ? probe_bucket(nbk0, R0, key, mask) : R0, i = R + o;
    uint32_t step = 0;   // order position of slot i within bucket R
    // at most one probe step per slot, and one retry per other touch of the
    // key in the batch (each failed retry means another touch got in)
    uint64_t limit = mask + 1 + (1ull << 20);
    if (loop_limit && loop_limit < limit) limit = loop_limit;
    for (uint64_t it = 0; it < limit; ++it) {
        if (old.key == 0) { *claimed = true; return 0; }   // a CAS from {0,0} that failed returns a key
        if (old.key == key) {   // the slot's key never changes: raise its position word alone
            if (old.pos1 >= p1) return old.pos1;
            return pos_max(&t[i], p1);
        }
        Slot sn[kGroup];
#pragma unroll
        for (int j = 0; j < (int)kGroup; ++j) sn[j] = load_slot(t + R + j);
        uint32_t best = kGroup;
        Slot bs{0, 0};
#pragma unroll
        for (int j = 0; j < (int)kGroup; ++j) {
            const uint32_t q = (uint32_t(j) - o) & (kGroup - 1);
            if ((sn[j].key == 0 || sn[j].key == key) && q > step && q < best) {
                best = q;
                bs = sn[j];
            }
        }
        if (best < kGroup) {
            step = best;
        } else {
            R = probe_bucket(++nbk, R0, key, mask);
            step = 0;
            bs = Slot{0, 0};
        }
        i = R + ((o + step) & (kGroup - 1));
        old = bs.key == key ? bs : slot_cas(&t[i], Slot{0, 0}, Slot{key, p1});
    }
    set_err(err, DM_ERR_TIMEOUT);
    return 0;
}

// Insert a key known to be absent (index rebuild: all keys distinct).
__device__ __forceinline__ void table_insert_new(Slot *t, uint64_t mask, uint64_t key, uint64_t home, uint64_t p1,
                                                 uint32_t *err) {
    bool cl = false;
    touch_resolve(t, mask, key, p1, home, slot_cas(&t[home], Slot{0, 0}, Slot{key, p1}), err, &cl);
}

// Point an existing key at a new record position (log compaction; no other
// thread touches the key meanwhile).
__device__ __forceinline__ void table_set_pos(Slot *t, uint64_t mask, uint64_t key, uint64_t home, uint64_t p1,
                                              uint32_t *err) {
    Slot s;
    const uint64_t j = table_find(t, mask, key, home, err, &s);
    if (j == kNoSlot) set_err(err, DM_ERR_TIMEOUT);
    else t[j].pos1 = p1;
}

// Exclusive block scan of u32 counts (any block size up to 1024).
__device__ __forceinline__ uint32_t block_excl_u32(uint32_t v, uint32_t *s_w, uint32_t &total) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    uint32_t inc = v;
#pragma unroll
    for (int dd = 1; dd < 32; dd <<= 1) {
        const uint32_t u = __shfl_up_sync(0xffffffffu, inc, dd);
        if (lane >= dd) inc += u;
    }
    if (lane == 31) s_w[wid] = inc;
    __syncthreads();
    if (wid == 0) {
        const uint32_t x = lane < (int)(blockDim.x >> 5) ? s_w[lane] : 0;
        uint32_t y = x;
#pragma unroll
        for (int dd = 1; dd < 32; dd <<= 1) {
            const uint32_t u = __shfl_up_sync(0xffffffffu, y, dd);
            if (lane >= dd) y += u;
        }
        s_w[lane] = y - x;
        if (lane == 31) s_w[32] = y;
    }
    __syncthreads();
    const uint32_t r = s_w[wid] + inc - v;
    total = s_w[32];
    __syncthreads();
    return r;
}

// Instance owning flat chunk c of a chunk-offset table (largest i with off[i] <= c).
__device__ __forceinline__ uint32_t owner_of(const uint32_t *off, uint32_t M, uint32_t c) {
    uint32_t lo = 0, hi = M;
    while (hi - lo > 1) {
        const uint32_t mid = (lo + hi) >> 1;
        if (off[mid] <= c) lo = mid; else hi = mid;
    }
    return lo;
}

// ---------------------------------------------------------------------------
// Maintenance before the touches.
//   plan  blocks each instance receives, which instances need a compaction
//         (log would overflow) or a rebuild (index would pass its rebuild
//         threshold),
//         and the chunk lists of both: every CTA of kernel a computes the
//         same plan from the same inputs in its shared memory, CTA 0 also
//         stores it for the kernels after;
//   a     grid: clear the second index (rebuild) / stale flags (compaction),
//         count live records per 1024-record chunk of the log; the last CTA
//         to finish turns the counts into destination offsets (a warp per
//         compacting instance);
//   c     grid: walk the live records; compaction copies them in order into
//         the second log (and repoints their index slots, or inserts them
//         into the second index when rebuilding too); a rebuild alone
//         inserts them with their current positions.  The last CTA to
//         finish (CTA 0 when there was nothing to walk) swaps the new logs
//         and indices in and lays out the commit's records.
// Kernels a and c do nothing else when the plan asks for no maintenance, the
// usual case; "last CTA" is an atomic count of finished CTAs, no CTA waits.

// The plan in shared memory (dynamic, plan_smem(M) bytes).
struct PlanSm {
    uint64_t *cnt;       // M: blocks each instance receives
    uint32_t *fl;        // M: kFlagCompact | kFlagRebuild
    uint32_t *mc, *mr;   // M + 1: chunk offsets of the log walk and of the clearing
    uint32_t *rk;        // M: pool slot of a rebuilding instance
};
__device__ __forceinline__ PlanSm plan_sm(unsigned char *smem, uint32_t M) {
    PlanSm p;
    p.cnt = reinterpret_cast<uint64_t *>(smem);
    p.fl = reinterpret_cast<uint32_t *>(p.cnt + M);
    p.mc = p.fl + M;
    p.mr = p.mc + M + 1;
    p.rk = p.mr + M + 1;
    return p;
}
static size_t plan_smem(uint32_t M) { return size_t(M) * 24 + 8; }

// The plan, computed by a whole CTA; `store`: also write it to global
// memory (flags, chunk offsets, pool slots and buffers, the rotation start
// the commit prep installs, the counters of this commit).
__device__ void maint_plan_cta(const DevState &d, uint32_t n, const PlanSm &P, bool store) {
    __shared__ uint32_t s_w[33];
    __shared__ uint32_t s_served, s_last;
    // blocks each instance receives: the choice kernel's count, unless a
    // rebalance has moved a request of the batch since
    const bool dirty = d.info->final_dirty != 0;
    for (uint32_t i = threadIdx.x; i < d.M; i += blockDim.x) P.cnt[i] = dirty ? 0 : d.log_adv[i];
    __syncthreads();
    for (uint32_t r0 = threadIdx.x; dirty && r0 < n; r0 += 4 * blockDim.x) {   // four loads in flight per thread
        uint32_t f[4], nb[4];
#pragma unroll
        for (uint32_t u = 0; u < 4; ++u) {
            const uint32_t r = r0 + u * blockDim.x;
            f[u] = r < n ? d.r_final[r] : 0;
            nb[u] = r < n ? d.r_nblk[r] : 0;
        }
#pragma unroll
        for (uint32_t u = 0; u < 4; ++u)
            if (nb[u]) atomicAdd(reinterpret_cast<unsigned long long *>(&P.cnt[f[u]]), (unsigned long long)nb[u]);
    }
    __syncthreads();
    // 1) what each instance needs: compaction if its log would overflow,
    //    a rebuild if its index would pass rb_thr taken slots
    for (uint32_t i = threadIdx.x; i < d.M; i += blockDim.x) {
        uint32_t fl = 0;
        if (d.table[i]) {
            const uint64_t cnt = P.cnt[i];
            if (cnt > d.T) set_err(d.err, DM_ERR_CAPACITY);
            if (d.log_tail[i] - d.log_front[i] + cnt > d.logcap) fl |= kFlagCompact;
            if (d.used[i] + cnt > d.rb_thr) fl |= kFlagRebuild;
        }
        P.fl[i] = fl;
    }
    if (threadIdx.x == 0) { s_served = 0; s_last = 0; }
    __syncthreads();
    // 2) rebuilds take spare buffers from the pool, in id order from a
    //    rotating start; those beyond the pool wait for a later commit (each
    //    waits at most ceil(M / pool) commits; dm_create checks the index
    //    has that much headroom above half full).  The new start is
    //    installed by the commit prep, after every CTA has read the old one.
    const uint32_t rr = *d.rb_rr;
    for (uint32_t base = 0; base < d.M; base += blockDim.x) {
        const uint32_t k = base + threadIdx.x;
        const uint32_t i = k < d.M ? (rr + k) % d.M : 0;
        const bool want = k < d.M && (P.fl[i] & kFlagRebuild);
        uint32_t tot;
        const uint32_t rank = s_served + block_excl_u32(want ? 1u : 0u, s_w, tot);
        if (want) {
            if (rank < d.pool_n) {
                P.rk[i] = rank;
                if (store) {
                    d.rb_slot[i] = rank;
                    d.table_alt[i] = d.pool[rank];
                }
                atomicMax(&s_last, k);   // the last position served
            } else {
                P.fl[i] &= ~kFlagRebuild;
            }
        }
        __syncthreads();
        if (threadIdx.x == 0) s_served += tot;
        __syncthreads();
    }
    if (store && threadIdx.x == 0) d.info->rb_rr_next = s_served ? (rr + s_last + 1) % d.M : rr;
    // 3) chunk offsets of the work the final flags ask for
    uint32_t cw = 0, cz = 0;
    for (uint32_t base = 0; base < d.M; base += blockDim.x) {
        const uint32_t i = base + threadIdx.x;
        uint32_t nw = 0, nz = 0, fl = 0;
        if (i < d.M && d.table[i]) {
            fl = P.fl[i];
            const uint64_t len = d.log_tail[i] - d.log_front[i];
            if (fl & kFlagCompact) nz += (uint32_t)((d.logcap + kZeroChunk - 1) / kZeroChunk);
            if (fl & kFlagRebuild) nz += (uint32_t)((d.S + kZeroChunk - 1) / kZeroChunk);
            if (fl) nw = (uint32_t)((len + kEvChunk - 1) / kEvChunk);
        }
        uint32_t tw, tz;
        const uint32_t ew = block_excl_u32(nw, s_w, tw);
        const uint32_t ez = block_excl_u32(nz, s_w, tz);
        if (i < d.M) {
            P.mc[i] = cw + ew;
            P.mr[i] = cz + ez;
            P.fl[i] = fl;
            if (store) {
                d.mc_chunk_off[i] = cw + ew;
                d.mr_chunk_off[i] = cz + ez;
                d.mt_flags[i] = fl;
            }
        }
        cw += tw;
        cz += tz;
    }
    if (threadIdx.x == 0) {
        P.mc[d.M] = cw;
        P.mr[d.M] = cz;
        if (store) {
            d.mc_chunk_off[d.M] = cw;
            d.mr_chunk_off[d.M] = cz;
            d.info->mc_chunks = cw;
            d.info->mr_chunks = cz;
            d.info->mt_done_c = 0;
            if (cw > d.mc_cap) set_err(d.err, DM_ERR_CAPACITY);
        }
    }
    __syncthreads();
}

// True in the one CTA of the grid that finishes last (count: a counter the
// plan kernel zeroed).  Called by all threads of every CTA that gets here.
__device__ __forceinline__ bool last_cta(uint32_t *count) {
    __shared__ uint32_t s_last;
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        s_last = atomicAdd(count, 1u) + 1 == gridDim.x;
    }
    __syncthreads();
    if (s_last) __threadfence();
    return s_last != 0;
}

// Warp per compacting instance: chunk counts -> exclusive destination
// offsets (the counts of other CTAs are read from L2).
__device__ void compact_scan_cta(const DevState &d, const PlanSm &P) {
    const int lane = threadIdx.x & 31;
    for (uint32_t i = threadIdx.x >> 5; i < d.M; i += blockDim.x >> 5) {
        if (!(P.fl[i] & kFlagCompact)) continue;
        const uint32_t c0 = P.mc[i], c1 = P.mc[i + 1];
        uint64_t carry = 0;
        for (uint32_t cb = c0; cb < c1; cb += 32) {
            const uint32_t c = cb + lane;
            const uint64_t v = c < c1 ? __ldcg(&d.mc_chunk_live[c]) : 0;
            const uint64_t inc = warp_incl_scan(v, lane);
            if (c < c1) d.mc_chunk_live[c] = (uint32_t)(carry + inc - v);
            carry += shfl_u64(inc, 31);
        }
        if (lane == 0) d.mt_newtail[i] = d.log_front[i] + carry;
    }
}

// n: requests of the batch; dynamic smem: plan_smem(M) bytes.
__global__ void __launch_bounds__(kMtThreads) k_maint_a(DevState d, uint32_t n) {
    pdl_enter();
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ uint32_t s_i, s_cnt[kMtThreads / 32];
    if (has_err(d.err)) return;
    const PlanSm P = plan_sm(smem, d.M);
    maint_plan_cta(d, n, P, blockIdx.x == 0);
    // clearing: a rebuilding instance's chunks cover its second index first,
    // a compacting instance's (then) its second stale-flag array
    const uint32_t nz = P.mr[d.M];
    for (uint32_t c = blockIdx.x; c < nz; c += gridDim.x) {
        if (threadIdx.x == 0) s_i = owner_of(P.mr, d.M, c);
        __syncthreads();
        const uint32_t i = s_i;
        const uint32_t fl = P.fl[i];
        uint64_t k = uint64_t(c - P.mr[i]) * kZeroChunk;
        const uint64_t tab = (fl & kFlagRebuild) ? d.S : 0;
        const uint64_t tab_chunks_end = (tab + kZeroChunk - 1) / kZeroChunk * kZeroChunk;
        if (k < tab_chunks_end) {
            Slot *t = d.pool[P.rk[i]];
            for (uint32_t q = threadIdx.x; q < kZeroChunk; q += kMtThreads)
                if (k + q < tab) t[k + q] = Slot{0, 0};
        } else {
            k -= tab_chunks_end;
            uint8_t *f = d.stale_alt[i];
            for (uint32_t q = threadIdx.x; q < kZeroChunk; q += kMtThreads)
                if (k + q < d.logcap) f[k + q] = 0;
        }
        __syncthreads();
    }
    // live records per log chunk of every instance being maintained (none
    // when the chunk list would not fit: the plan has recorded the error)
    const uint32_t nw = P.mc[d.M] <= d.mc_cap ? P.mc[d.M] : 0;
    const uint64_t lmask = d.logcap - 1;
    for (uint32_t c = blockIdx.x; c < nw; c += gridDim.x) {
        if (threadIdx.x == 0) s_i = owner_of(P.mc, d.M, c);
        __syncthreads();
        const uint32_t i = s_i;
        const uint64_t tail = d.log_tail[i];
        const uint64_t base = d.log_front[i] + uint64_t(c - P.mc[i]) * kEvChunk;
        const uint8_t *st = d.stale[i];
        uint32_t cnt = 0;
        for (uint32_t k = threadIdx.x; k < kEvChunk; k += kMtThreads)
            cnt += (base + k < tail && !st[(base + k) & lmask]);
        cnt = __reduce_add_sync(0xffffffffu, cnt);
        if ((threadIdx.x & 31) == 0) s_cnt[threadIdx.x >> 5] = cnt;
        __syncthreads();
        if (threadIdx.x == 0) {
            uint32_t t = 0;
            for (int w = 0; w < kMtThreads / 32; ++w) t += s_cnt[w];
            d.mc_chunk_live[c] = t;
        }
        __syncthreads();
    }
    if (nw && last_cta(&d.info->mt_done_a)) {
        compact_scan_cta(d, P);
        if (threadIdx.x == 0) d.info->mt_done_a = 0;   // for the next commit
    }
}

__device__ void commit_prep_cta(const DevState &d, uint32_t n, uint64_t *adv);

// n: requests of the batch (for the record layout); dynamic smem: one u64
// per instance.
__global__ void __launch_bounds__(kMtThreads) k_maint_c(DevState d, uint32_t n) {
    pdl_enter();
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ uint32_t s_i, s_w[kMtThreads / 32];
    if (has_err(d.err)) return;
    const uint32_t nw = d.info->mc_chunks;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const uint64_t lmask = d.logcap - 1, mask = d.S - 1;
    for (uint32_t c = blockIdx.x; c < nw; c += gridDim.x) {
        if (threadIdx.x == 0) s_i = owner_of(d.mc_chunk_off, d.M, c);
        __syncthreads();
        const uint32_t i = s_i;
        const uint32_t fl = d.mt_flags[i];
        const uint64_t front = d.log_front[i], tail = d.log_tail[i];
        const uint64_t base = front + uint64_t(c - d.mc_chunk_off[i]) * kEvChunk;
        const Rec *lg = d.logbuf[i];
        const uint8_t *st = d.stale[i];
        uint64_t out = front + ((fl & kFlagCompact) ? d.mc_chunk_live[c] : 0);
        for (uint32_t k0 = 0; k0 < kEvChunk; k0 += kMtThreads) {   // keeps record order
            const uint64_t p = base + k0 + threadIdx.x;
            const bool live = p < tail && !st[p & lmask];
            const uint32_t b = __ballot_sync(0xffffffffu, live);
            if (lane == 0) s_w[wid] = __popc(b);
            __syncthreads();
            uint32_t before = 0, tot = 0;
            for (int w = 0; w < kMtThreads / 32; ++w) {
                before += w < wid ? s_w[w] : 0;
                tot += s_w[w];
            }
            if (live) {
                const Rec r = lg[p & lmask];
                const uint32_t home = d.loghome[i][p & lmask];
                if (fl & kFlagCompact) {
                    const uint64_t np = out + before + __popc(b & ((1u << lane) - 1));
                    d.logbuf_alt[i][np & lmask] = r;
                    d.loghome_alt[i][np & lmask] = home;
                    if (fl & kFlagRebuild) table_insert_new(d.table_alt[i], mask, r.key, home, np + 1, d.err);
                    else table_set_pos(d.table[i], mask, r.key, home, np + 1, d.err);
                } else {
                    table_insert_new(d.table_alt[i], mask, r.key, home, p + 1, d.err);
                }
            }
            out += tot;
            __syncthreads();
        }
    }
    if (nw ? last_cta(&d.info->mt_done_c) : blockIdx.x == 0)
        commit_prep_cta(d, n, reinterpret_cast<uint64_t *>(smem));
}

// ---------------------------------------------------------------------------
// Swap in compacted logs / rebuilt indices, fix each instance's log base for
// this commit and advance its tail.  The choice kernel already placed every
// request among its instance's records; only when a rebalance moved a
// request of this batch are the offsets recomputed (arrival order per final
// instance).  One CTA, after every CTA of k_maint_c; adv: one u64 per
// instance in shared memory.
__device__ void commit_prep_cta(const DevState &d, uint32_t n, uint64_t *adv) {
    __shared__ uint32_t s_f[kPrepChunk], s_nb[kPrepChunk];
    __shared__ uint64_t s_off[kPrepChunk];
    for (uint32_t i = threadIdx.x; i < d.M; i += blockDim.x) {
        const uint32_t fl = d.mt_flags[i];
        if (fl & kFlagCompact) {
            Rec *a = d.logbuf[i];
            d.logbuf[i] = d.logbuf_alt[i];
            d.logbuf_alt[i] = a;
            uint8_t *f = d.stale[i];
            d.stale[i] = d.stale_alt[i];
            d.stale_alt[i] = f;
            uint32_t *hm = d.loghome[i];
            d.loghome[i] = d.loghome_alt[i];
            d.loghome_alt[i] = hm;
            d.log_tail[i] = d.mt_newtail[i];
            atomicAdd(reinterpret_cast<unsigned long long *>(&d.maint_count[1]), 1ull);
        }
        if (fl & kFlagRebuild) {   // the old index goes back to the pool
            d.pool[d.rb_slot[i]] = d.table[i];
            d.table[i] = d.table_alt[i];
            d.table_alt[i] = nullptr;
            d.used[i] = d.live[i];
            atomicAdd(reinterpret_cast<unsigned long long *>(&d.maint_count[0]), 1ull);
        }
        adv[i] = d.log_adv[i];
    }
    const bool dirty = d.info->final_dirty != 0;
    if (dirty) {
        __syncthreads();
        for (uint32_t i = threadIdx.x; i < d.M; i += blockDim.x) adv[i] = 0;
        for (uint32_t base = 0; base < n; base += kPrepChunk) {
            const uint32_t m = min(kPrepChunk, n - base);
            __syncthreads();
            for (uint32_t k = threadIdx.x; k < m; k += blockDim.x) {
                s_f[k] = d.r_final[base + k];
                s_nb[k] = d.r_nblk[base + k];
            }
            __syncthreads();
            if (threadIdx.x == 0)
                for (uint32_t k = 0; k < m; ++k) {
                    const uint32_t f = s_f[k];
                    const uint64_t o = adv[f];
                    s_off[k] = o;
                    adv[f] = o + s_nb[k];
                }
            __syncthreads();
            for (uint32_t k = threadIdx.x; k < m; k += blockDim.x) d.r_touchoff[base + k] = s_off[k];
        }
        __syncthreads();
    }
    for (uint32_t i = threadIdx.x; i < d.M; i += blockDim.x) {
        const uint64_t b = d.log_tail[i];
        d.log_base[i] = b;
        d.log_tail[i] = b + adv[i];
    }
    if (threadIdx.x == 0) {
        d.info->clock_base = *d.clock;
        *d.clock += d.info->total_blocks;
        *d.rb_rr = d.info->rb_rr_next;
    }
}

// Index touches.  A superseded record (the key's previous record, or this
// one when a later touch of the batch already won) gets its stale flag.
__device__ __forceinline__ void touch_outcome(uint64_t old, uint64_t p, uint64_t front, uint8_t *st, uint64_t lmask,
                                              uint32_t &newly) {
    if (old == 0 || old - 1 < front) {
        ++newly;                                  // new or evicted: resident again
    } else if (old - 1 < p) {
        st[(old - 1) & lmask] = 1;                // previous record superseded
    } else {
        st[p & lmask] = 1;                        // a later touch of this batch won
    }
}

// Per-segment values of the touch kernel.  Within a segment, block e
// (0..cnt-1) has log position p_first - e and stamp stamp_first - e: a
// request touches its blocks from the last one down.
struct TouchSeg {
    uint64_t pidx;          // plocal index of the segment's first block
    uint64_t p_first;       // log position of that block's record
    uint64_t stamp_first;   // its clock stamp
    uint64_t carry;         // prefix carry into the segment
    uint64_t front;         // log front of the final instance
    Slot *t;
    Rec *lg;
    uint8_t *st;
    uint32_t *lh;           // index home of each record
    uint32_t cnt, f;        // blocks in the segment, final instance
    uint64_t kpos;          // DM_REBALANCE_FRESH_HITS: ring position of its first block's key on f
};

__device__ __forceinline__ TouchSeg touch_seg_load(const DevState &d, uint32_t seg, uint64_t clock_base) {
    const uint32_t r = d.seg_req[seg];
    const uint32_t first = (seg - d.r_segoff[r]) * kSegBlocks;
    const uint32_t nblk = d.r_nblk[r], f = d.r_final[r];
    const uint64_t bo = d.r_blkoff[r];
    TouchSeg g;
    g.pidx = bo + first;
    g.p_first = d.log_base[f] + d.r_touchoff[r] + (nblk - 1 - first);
    g.stamp_first = clock_base + bo + (nblk - first);
    g.carry = d.seg_carry[seg];
    g.front = d.log_front[f];
    g.t = d.table[f];
    g.lg = d.logbuf[f];
    g.st = d.stale[f];
    g.lh = d.loghome[f];
    g.cnt = min(nblk - first, kSegBlocks);
    g.f = f;
    g.kpos = d.KQ ? d.r_koff[r] + first : 0;
    // the segment's records lie inside the instance's log window
    DM_CHECK(f < d.M && g.p_first + 1 - g.front <= d.logcap && g.pidx + g.cnt <= d.max_blocks, d.err);
    return g;
}

// Each warp takes a contiguous range of segments.  Its lanes load the
// metadata of up to 32 of them at once into the warp's shared-memory slots
// (request, final instance, offsets: one dependent chain per 32 segments
// instead of per segment); then, segment by segment, lane l touches blocks l
// and l+32: both home-slot CAS are issued before either result is used, and
// the next segment's plocal values are loaded while they are in flight.
// Touches that one or two atomics did not settle are deferred to the end of
// the 32 segments, where the warp's lanes take them one each, whatever their
// segment, and walk the key's probe order (touch_resolve: a CAS claim or a
// position max, concurrent with every other touch of the key, so the order
// in which warps get there does not matter).  No CTA barriers: a warp never
// waits for another.
constexpr int kTouchThreads = 256;
__global__ void __launch_bounds__(kTouchThreads, 4) k_commit_touch(DevState d) {
    pdl_enter();
    __shared__ TouchSeg s_seg[kTouchThreads / 32][32];
    __shared__ uint32_t s_add[kTouchThreads / 32][2][32];   // deferred outcomes per segment: newly, claims
    if (has_err(d.err)) return;
    const int lane = threadIdx.x & 31;
    const uint32_t nw = (gridDim.x * blockDim.x) >> 5;
    const uint32_t gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint32_t total_segs = d.info->total_segs;
    const uint64_t clock_base = d.info->clock_base;
    const uint64_t mask = d.S - 1, lmask = d.logcap - 1;
    const uint32_t per = (total_segs + nw - 1) / nw;
    const uint32_t lo = min(total_segs, gw * per), hi = min(total_segs, lo + per);
    for (uint32_t c0 = lo; c0 < hi; c0 += 32) {
        const uint32_t nc = min(32u, hi - c0);
        TouchSeg *sg = s_seg[threadIdx.x >> 5];
        if ((uint32_t)lane < nc) sg[lane] = touch_seg_load(d, c0 + lane, clock_base);
        __syncwarp();
        uint32_t my_newly = 0, my_claims = 0, my_nd = 0;   // lane l: segment c0 + l
        uint64_t x0 = lane < (int)sg[0].cnt ? d.plocal[sg[0].pidx + lane] : 0;
        uint64_t x1 = lane + 32 < (int)sg[0].cnt ? d.plocal[sg[0].pidx + lane + 32] : 0;
        for (uint32_t i = 0; i < nc; ++i) {
            const TouchSeg &g = sg[i];
            const bool v0 = lane < (int)g.cnt, v1 = lane + 32 < (int)g.cnt;
            const uint64_t k0 = cache_key(x0 + g.carry, d.Sc), k1 = cache_key(x1 + g.carry, d.Sc);
            const uint64_t h0 = group_home(group_anchor(k0, lane), lane, mask);   // segments start on a group boundary
            const uint64_t h1 = group_home(group_anchor(k1, lane), lane, mask);
            const uint64_t p0 = g.p_first - lane, p1 = g.p_first - lane - 32;
            if (v0) {
                g.lg[p0 & lmask] = Rec{k0, g.stamp_first - lane};
                g.lh[p0 & lmask] = (uint32_t)h0;
            }
            if (v1) {
                g.lg[p1 & lmask] = Rec{k1, g.stamp_first - lane - 32};
                g.lh[p1 & lmask] = (uint32_t)h1;
            }
            if (d.KQ) {   // the queued request's keys, for fresh rebalancing probes
                uint64_t *kr = d.kring + uint64_t(g.f) * d.KQ;
                if (v0) kr[(g.kpos + lane) & (d.KQ - 1)] = k0;
                if (v1) kr[(g.kpos + lane + 32) & (d.KQ - 1)] = k1;
            }
            const Slot c0s = v0 ? slot_cas(&g.t[h0], Slot{0, 0}, Slot{k0, p0 + 1}) : Slot{0, 0};
            const Slot c1s = v1 ? slot_cas(&g.t[h1], Slot{0, 0}, Slot{k1, p1 + 1}) : Slot{0, 0};
            if (i + 1 < nc) {   // next segment's blocks, loaded while the CAS are in flight
                const uint64_t pi = sg[i + 1].pidx;
                const uint32_t cn = sg[i + 1].cnt;
                x0 = lane < (int)cn ? d.plocal[pi + lane] : 0;
                x1 = lane + 32 < (int)cn ? d.plocal[pi + lane + 32] : 0;
            }
            // a key found at its home with an older position: raised here by
            // an atomic max on its position word, which always settles the
            // touch (the value it returns orders it against every other
            // touch of the key).  A key whose home slot holds another key, in a
            // group whose 8 lanes found every slot of the home bucket taken
            // and none holding the key, continues its probe order in the
            // next bucket: one attempt there.  (Slots never empty again, so
            // the key can never belong to that bucket.)  All these attempts
            // are in flight together.
            Slot r0 = c0s, r1 = c1s;
            const bool up0 = v0 && c0s.key == k0 && c0s.pos1 <= p0;
            const bool up1 = v1 && c1s.key == k1 && c1s.pos1 <= p1;
            bool mv0, mv1;
            {
                const int gbase = lane & ~(int)(kGroup - 1), me = lane & (int)(kGroup - 1);
                const bool full0 = __shfl_sync(0xffffffffu, (int)v0, gbase + (int)kGroup - 1) != 0;
                const bool full1 = __shfl_sync(0xffffffffu, (int)v1, gbase + (int)kGroup - 1) != 0;
                const uint64_t seen0 = c0s.key == 0 ? k0 : c0s.key, seen1 = c1s.key == 0 ? k1 : c1s.key;
                bool in0 = false, in1 = false;
#pragma unroll
                for (int j = 0; j < (int)kGroup; ++j) {
                    const uint64_t s0 = shfl_u64(seen0, gbase + j), s1 = shfl_u64(seen1, gbase + j);
                    in0 |= j != me && s0 == k0;
                    in1 |= j != me && s1 == k1;
                }
                mv0 = v0 && full0 && c0s.key != 0 && c0s.key != k0 && !in0;
                mv1 = v1 && full1 && c1s.key != 0 && c1s.key != k1 && !in1;
            }
            const uint64_t n0 = probe_bucket(1, h0 & ~uint64_t(kGroup - 1), k0, mask) | (h0 & (kGroup - 1));
            const uint64_t n1 = probe_bucket(1, h1 & ~uint64_t(kGroup - 1), k1, mask) | (h1 & (kGroup - 1));
            if (up0) r0 = Slot{k0, pos_max(&g.t[h0], p0 + 1)};
            else if (mv0) r0 = slot_cas(&g.t[n0], Slot{0, 0}, Slot{k0, p0 + 1});
            if (up1) r1 = Slot{k1, pos_max(&g.t[h1], p1 + 1)};
            else if (mv1) r1 = slot_cas(&g.t[n1], Slot{0, 0}, Slot{k1, p1 + 1});
            // settled here: a claim of an empty home slot, a raise that went
            // through, or the key found with a later position already; the
            // rest is deferred (x: the position value seen last)
            uint32_t newly = 0, claims = 0;
            bool need0 = false, need1 = false;
            uint64_t x0 = c0s.pos1, x1 = c1s.pos1;
            if (v0) {
                if (c0s.key == 0 || (mv0 && r0.key == 0)) { ++newly; ++claims; }
                else if (mv0 && r0.key == k0 && r0.pos1 > p0) touch_outcome(r0.pos1, p0, g.front, g.st, lmask, newly);
                else if (mv0) { need0 = true; x0 = r0.pos1; }
                else if (up0) touch_outcome(r0.pos1, p0, g.front, g.st, lmask, newly);   // the max settles it
                else if (!up0 && c0s.key == k0) touch_outcome(c0s.pos1, p0, g.front, g.st, lmask, newly);
                else { need0 = true; x0 = c0s.pos1; }
            }
            if (v1) {
                if (c1s.key == 0 || (mv1 && r1.key == 0)) { ++newly; ++claims; }
                else if (mv1 && r1.key == k1 && r1.pos1 > p1) touch_outcome(r1.pos1, p1, g.front, g.st, lmask, newly);
                else if (mv1) { need1 = true; x1 = r1.pos1; }
                else if (up1) touch_outcome(r1.pos1, p1, g.front, g.st, lmask, newly);
                else if (!up1 && c1s.key == k1) touch_outcome(c1s.pos1, p1, g.front, g.st, lmask, newly);
                else { need1 = true; x1 = c1s.pos1; }
            }
            // deferred touches go to the segment's own slice of the queue
            const uint32_t m0 = __ballot_sync(0xffffffffu, need0), m1 = __ballot_sync(0xffffffffu, need1);
            const uint32_t below = (1u << lane) - 1u;
            Deferred *dq = d.defer + uint64_t(c0 + i) * kSegBlocks;
            // found: the key sits at the preferred slot of the recorded bucket
            // (its home, or the next bucket after a move) with position x
            if (need0)
                dq[__popc(m0 & below)] = Deferred{k0, p0, x0, (uint32_t)h0,
                                                  (uint16_t)((mv0 ? r0.key : c0s.key) == k0), (uint16_t)mv0};
            if (need1)
                dq[__popc(m0) + __popc(m1 & below)] = Deferred{k1, p1, x1, (uint32_t)h1,
                                                               (uint16_t)((mv1 ? r1.key : c1s.key) == k1),
                                                               (uint16_t)mv1};
            newly = __reduce_add_sync(0xffffffffu, newly);
            claims = __reduce_add_sync(0xffffffffu, claims);
            if (lane == (int)i) {
                my_newly = newly;
                my_claims = claims;
                my_nd = __popc(m0) + __popc(m1);
            }
        }
        if (__ballot_sync(0xffffffffu, my_nd != 0)) {
            // the deferred touches of these segments, numbered segment by
            // segment: lane l takes touch e0 + l
            uint32_t *add_n = s_add[threadIdx.x >> 5][0], *add_c = s_add[threadIdx.x >> 5][1];
            add_n[lane] = 0;
            add_c[lane] = 0;
            uint32_t incl = my_nd;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t u = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += u;
            }
            const uint32_t excl = incl - my_nd, E = __shfl_sync(0xffffffffu, incl, 31);
            __syncwarp();
            for (uint32_t e0 = 0; e0 < E; e0 += 32) {
                const uint32_t e = e0 + lane;
                uint32_t sj = 0;   // its segment: the number of segments whose touches end at or before e
#pragma unroll
                for (uint32_t step = 16; step; step >>= 1)
                    if (__shfl_sync(0xffffffffu, incl, sj + step - 1) <= e) sj += step;
                const uint32_t first = __shfl_sync(0xffffffffu, excl, sj);
                if (e < E) {
                    const TouchSeg &g = sg[sj];
                    const Deferred en = d.defer[uint64_t(c0 + sj) * kSegBlocks + (e - first)];
                    // the slot as the touch saw it last (another key: any value
                    // other than 0 and the key)
                    const Slot old = en.found ? Slot{en.key, en.x} : Slot{en.key == 1 ? 2ull : en.key ^ 1ull, 0};
                    bool cl = false;
                    uint32_t nw = 0;
                    const uint64_t o = touch_resolve(g.t, mask, en.key, en.p + 1, en.home, old, d.err, &cl,
                                                     en.bucket, d.loop_limit);
                    touch_outcome(o, en.p, g.front, g.st, lmask, nw);
                    if (nw) atomicAdd(&add_n[sj], nw);
                    if (cl) atomicAdd(&add_c[sj], 1u);
                }
            }
            __syncwarp();
            my_newly += add_n[lane];
            my_claims += add_c[lane];
        }
        {   // keys made resident and index slots taken, per final instance:
            // one atomic per instance for these 32 segments (mostly of one request)
            const uint32_t fi = (uint32_t)lane < nc ? sg[lane].f : 0xffffffffu;
            const uint32_t peers = __match_any_sync(0xffffffffu, fi);
            const uint32_t sa = __reduce_add_sync(peers, my_newly), sb = __reduce_add_sync(peers, my_claims);
            if ((uint32_t)lane < nc && lane == __ffs(peers) - 1) {
                if (sa) atomicAdd(reinterpret_cast<unsigned long long *>(&d.live[fi]), (unsigned long long)sa);
                if (sb) atomicAdd(reinterpret_cast<unsigned long long *>(&d.used[fi]), (unsigned long long)sb);
            }
        }
        __syncwarp();   // the slots are refilled for the next 32 segments
    }
}

// ---------------------------------------------------------------------------
// Eviction.  Instance i drops its excess_i = live_i - C oldest resident keys
// by moving its log front just past the excess_i-th non-stale record; the
// stale flags it passes are reset (those positions will hold new records).
// A cluster of CTAs walks an instance's log from the front (k_evict below);
// the touch kernel has added the batch's newly resident keys to live_i.

constexpr int kEvThreads = 512;
constexpr uint32_t kEvCluster = 4;                                // CTAs sharing one instance's walk
constexpr uint32_t kEvVec = 4;                                    // 16-byte flag loads per thread and round, at most
constexpr uint32_t kEvPer = 16 * kEvVec;                          // records per thread and round, at most

// A cluster of kEvCluster CTAs per instance (persistent: clusters loop over
// instances).  Per round each CTA counts the non-stale records of its own
// span and posts the count in shared memory; after one cluster barrier every
// CTA reads all counts (distributed shared memory) and knows whether its
// span lies wholly before the cut (reset all its flags), holds it (find the
// exact record, reset up to it, write the new front) or lies after it.  The
// posted counts alternate between two slots, so one barrier per round
// suffices: a CTA cannot rewrite a slot before every CTA has passed the next
// barrier, which it reaches only after reading that slot.
__global__ void __cluster_dims__(kEvCluster, 1, 1) __launch_bounds__(kEvThreads) k_evict(DevState d) {
    pdl_enter();
    cg::cluster_group cluster = cg::this_cluster();
    __shared__ uint32_t s_w[33];
    __shared__ uint32_t s_tot[2], s_go;
    __shared__ uint64_t s_cut;
    __shared__ uint32_t s_ev[kMaxInstances];   // instances over capacity
    const uint32_t r = cluster.block_rank();
    const uint32_t cid = blockIdx.x / kEvCluster, ncl = gridDim.x / kEvCluster;
    // one decision for the whole cluster (rank 0's view of the error word)
    if (threadIdx.x == 0) s_go = !has_err(d.err);
    cluster.sync();
    const uint32_t go = *cluster.map_shared_rank(&s_go, 0);
    const uint64_t lmask = d.logcap - 1;
    uint32_t slot = 0;
    // the instances over capacity, in id order (every CTA builds the same
    // list), dealt to the clusters in turn
    uint32_t nev = 0;
    for (uint32_t base = 0; go && base < d.M; base += blockDim.x) {
        const uint32_t i = base + threadIdx.x;
        const bool over = i < d.M && d.table[i] && d.live[i] > d.C;
        uint32_t tot;
        const uint32_t rk = block_excl_u32(over ? 1u : 0u, s_w, tot);
        if (over) s_ev[nev + rk] = i;
        nev += tot;
    }
    __syncthreads();
    for (uint32_t e = cid; go && e < nev; e += ncl) {
        const uint32_t i = s_ev[e];
        uint64_t remaining = d.live[i] - d.C;
        uint8_t *st = d.stale[i];
        const uint64_t tail = d.log_tail[i];
        const uint64_t front0 = d.log_front[i];
        uint64_t front = front0;
        // rounds start on kEvPer-record boundaries (flags are read 16 at a
        // time; logcap is a power of two >= kEvPer); records before the
        // front in the first round do not count
        uint64_t base = front & ~uint64_t(kEvPer - 1);
        for (uint64_t it = 0; remaining > 0 && base < tail && it < kSpinLimit; ++it) {
            // a round reads about twice the records still to evict (stale
            // ones lie between them), 1-4 flag vectors per thread; the
            // choice depends on `remaining` alone, the same in every CTA
            const uint64_t vspan = uint64_t(kEvThreads) * kEvCluster * 16;
            const uint64_t want = (2 * remaining + vspan - 1) / vspan;
            const uint32_t vec = want >= kEvVec ? kEvVec : (want < 1 ? 1u : (uint32_t)want);
            const uint32_t per = 16 * vec;
            const uint64_t p0 = base + r * (uint64_t(kEvThreads) * per) + uint64_t(threadIdx.x) * per;
            // records [lo, hi) of the thread's `per` are after the front and before the tail
            const uint32_t lo = front > p0 ? (uint32_t)min(front - p0, (uint64_t)per) : 0u;
            const uint32_t hi = tail > p0 ? (uint32_t)min(tail - p0, (uint64_t)per) : 0u;
            uint64_t live_bits = 0;
#pragma unroll
            for (uint32_t k = 0; k < kEvVec; ++k) {
                if (k >= vec || 16 * k >= hi) continue;
                const uint4 v = *reinterpret_cast<const uint4 *>(st + ((p0 + 16 * k) & lmask));
                const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    // bit j of the nibble: flag byte j of the word is 0
                    const uint32_t z = __vcmpeq4(w[q], 0u) & 0x01010101u;
                    live_bits |= uint64_t((z * 0x10204080u) >> 28) << (16 * k + 4 * q);
                }
            }
            const uint64_t below_hi = hi >= 64 ? ~0ull : (1ull << hi) - 1;
            const uint64_t below_lo = lo >= 64 ? ~0ull : (1ull << lo) - 1;
            live_bits &= below_hi & ~below_lo;
            const uint32_t cnt = __popcll(live_bits);
            uint32_t tot;
            const uint32_t ex = block_excl_u32(cnt, s_w, tot);
            if (threadIdx.x == 0) s_tot[slot] = tot;
            cluster.sync();   // every span's count is visible
            uint64_t pre = 0, all = 0;
#pragma unroll
            for (uint32_t q = 0; q < kEvCluster; ++q) {
                const uint32_t t = *cluster.map_shared_rank(&s_tot[slot], q);
                pre += q < r ? t : 0;
                all += t;
            }
            slot ^= 1;
            // end of the records this span evicts: all of them, up to the
            // cut, or none
            uint64_t cut;
            if (pre + tot < remaining) {
                cut = ~0ull;
            } else if (pre < remaining) {
                const uint64_t need = remaining - pre;
                if (threadIdx.x == 0) s_cut = ~0ull;
                __syncthreads();
                if (ex < need && need <= ex + cnt) {   // exactly one thread
                    const uint32_t lw = (uint32_t)live_bits, nlo = __popc(lw);
                    const uint32_t m = (uint32_t)(need - ex);
                    const uint32_t bit =
                        m <= nlo ? __fns(lw, 0, (int)m) : 32 + __fns((uint32_t)(live_bits >> 32), 0, (int)(m - nlo));
                    s_cut = p0 + bit + 1;
                }
                __syncthreads();
                cut = s_cut;
                if (threadIdx.x == 0) d.log_front[i] = cut;
            } else {
                cut = 0;
            }
            // reset the flags of the records the front passes: [lo, b) of the thread's
            {
                const uint32_t b = cut > p0 ? (uint32_t)min(cut - p0, (uint64_t)hi) : 0u;
#pragma unroll
                for (uint32_t k = 0; k < kEvVec; ++k) {
                    const uint32_t k0 = 16 * k, k1 = k0 + 16;
                    if (k1 <= lo || k0 >= b) continue;
                    uint8_t *f = st + ((p0 + k0) & lmask);
                    if (lo <= k0 && k1 <= b) {
                        *reinterpret_cast<uint4 *>(f) = make_uint4(0, 0, 0, 0);
                    } else {
                        for (uint32_t q = max(lo, k0); q < min(b, k1); ++q) f[q - k0] = 0;
                    }
                }
            }
            remaining -= min(remaining, all);
            base += uint64_t(kEvThreads) * per * kEvCluster;
            front = min(base, tail);
        }
        if (r == 0 && threadIdx.x == 0) {
            if (remaining) {   // the log must cover every live key
                set_err(d.err, DM_ERR_TIMEOUT);
                d.log_front[i] = front;
            }
            d.live[i] = d.C;
        }
    }
    cluster.sync();   // no CTA leaves while another may still read its shared memory
}

// Clusters of the eviction kernel that can be resident at once (CTAs).
static int evict_grid() {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(kEvCluster);
    cfg.blockDim = dim3(kEvThreads);
    cudaLaunchAttribute at{};
    at.id = cudaLaunchAttributeClusterDimension;
    at.val.clusterDim.x = kEvCluster;
    at.val.clusterDim.y = 1;
    at.val.clusterDim.z = 1;
    cfg.attrs = &at;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, k_evict, &cfg) != cudaSuccess || n < 1) {
        cudaGetLastError();
        n = 1;
    }
    return n * (int)kEvCluster;
}

cudaError_t launch_commit(const DevState &d, uint32_t n, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    const size_t smem_a = plan_smem(d.M), smem_c = sizeof(uint64_t) * d.M;
    static size_t configured = 0;
    if (smem_a > configured) {   // smem_a > smem_c
        cudaError_t e = cudaFuncSetAttribute(k_maint_a, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_a);
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(k_maint_c, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_c);
        if (e != cudaSuccess) return e;
        configured = smem_a;
    }
    // every CTA of k_maint_a reads the whole batch for its plan: two per SM
    static const int g_a = full_grid(k_maint_a, kMtThreads) < 2 * sm_count() ? full_grid(k_maint_a, kMtThreads)
                                                                                : 2 * sm_count(),
                     g_c = full_grid(k_maint_c, kMtThreads), g_t = full_grid(k_commit_touch, kTouchThreads),
                     g_ev = evict_grid();
    DM_TRY(launch_pdl(k_maint_a, g_a, kMtThreads, smem_a, st, d, n));
    DM_TRY(launch_pdl(k_maint_c, g_c, kMtThreads, smem_c, st, d, n));
    DM_TRY(launch_pdl(k_commit_touch, g_t, kTouchThreads, 0, st, d));
    DM_TRY(launch_pdl(k_evict, g_ev, kEvThreads, 0, st, d));
    return cudaGetLastError();
}

}  // namespace dm
