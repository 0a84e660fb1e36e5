// dm_commit.cu -- cache save with exact LRU eviction (App. A.3.2 "KV cache
// save"; each instance keeps a bounded index of cached prefix blocks).
//
// Sequential definition: in arrival order, each request of the batch touches
// its block keys on its final instance from block n_blk-1 down to 0, one
// global clock tick per touch, and an LRU of capacity C evicts on overflow.
// An LRU holds exactly the C distinct keys with the latest last touch, so the
// GPU applies all touches of the batch at once (slot stamp = atomicMax of the
// touch stamps) and then evicts each instance's oldest keys down to C.
//
// Every instance keeps a recency log: the (key, stamp) of every touch in
// stamp order.  A log record is live when its stamp is still the key's slot
// stamp; evicting the k oldest keys = zeroing the slots of the first k live
// records from the log front.  Stale records are dropped by compaction, and
// the index (whose evicted keys keep their slots) is rebuilt from the
// compacted log when too many slots are used.
#include "dm_internal.cuh"

namespace dm {

// Touch key with stamp in an index: claims an empty slot for a new key, and
// raises the stamp to the newest touch.  Returns true when the key becomes
// resident (new, or previously evicted); *claimed when a slot was taken.
__device__ __forceinline__ bool table_touch(Slot *t, uint64_t mask, uint64_t key, uint64_t stamp,
                                            uint32_t *err, bool *claimed) {
    uint64_t i = key & mask;
    for (uint64_t it = 0; it <= mask; ++it) {
        uint64_t k = *(volatile uint64_t *)&t[i].key;
        if (k == 0) {
            const unsigned long long prev =
                atomicCAS(reinterpret_cast<unsigned long long *>(&t[i].key), 0ull, (unsigned long long)key);
            if (prev == 0) { *claimed = true; k = key; } else { k = prev; }
        }
        if (k == key) {
            const unsigned long long old =
                atomicMax(reinterpret_cast<unsigned long long *>(&t[i].stamp), (unsigned long long)stamp);
            return old == 0;
        }
        i = (i + 1) & mask;
    }
    set_err(err, DM_ERR_TIMEOUT);
    return false;
}

// Blocks each instance receives from the pending batch.
__global__ void k_commit_count(DevState d, uint32_t n) {
    if (has_err(d.err)) return;
    const uint32_t r = blockIdx.x * blockDim.x + threadIdx.x;
    if (r < n) atomicAdd(reinterpret_cast<unsigned long long *>(&d.touch_cnt[d.r_final[r]]),
                         (unsigned long long)d.r_nblk[r]);
}

// Block-wide exclusive scan of 0/1 flags (blockDim.x == 1024).
__device__ __forceinline__ uint32_t block_rank(bool f, uint32_t *s_w, uint32_t &total) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const uint32_t b = __ballot_sync(0xffffffffu, f);
    const uint32_t before = __popc(b & ((1u << lane) - 1));
    if (lane == 0) s_w[wid] = __popc(b);
    __syncthreads();
    if (wid == 0) {
        const uint32_t v = lane < (int)(blockDim.x >> 5) ? s_w[lane] : 0;
        uint32_t inc = v;
#pragma unroll
        for (int dd = 1; dd < 32; dd <<= 1) {
            const uint32_t u = __shfl_up_sync(0xffffffffu, inc, dd);
            if (lane >= dd) inc += u;
        }
        s_w[lane] = inc - v;
        if (lane == 31) s_w[32] = inc;
    }
    __syncthreads();
    const uint32_t r = s_w[wid] + before;
    total = s_w[32];
    __syncthreads();
    return r;
}

// Make room for the pending batch: compact an instance's log when it would
// overflow, rebuild its index when too many slots are used.  CTA per id.
__global__ void __launch_bounds__(1024) k_maintain(DevState d) {
    __shared__ uint32_t s_w[33];
    if (has_err(d.err)) return;
    const uint32_t i = blockIdx.x;
    Slot *t = d.table[i];
    if (!t) return;
    const uint64_t cnt = d.touch_cnt[i];
    if (cnt > d.T) {
        if (threadIdx.x == 0) set_err(d.err, DM_ERR_CAPACITY);
        return;
    }
    const uint64_t front = d.log_front[i], tail = d.log_tail[i];
    const bool rebuild = d.used[i] + cnt > d.S - d.S / 4;
    const bool compact = rebuild || (tail - front) + cnt > d.logcap;
    if (!compact) return;
    Slot *lg = d.logbuf[i];
    const uint64_t mask = d.S - 1, lmask = d.logcap - 1;
    uint64_t w = front;
    for (uint64_t p0 = front; p0 < tail; p0 += blockDim.x) {
        const uint64_t p = p0 + threadIdx.x;
        Slot e{0, 0};
        bool live = false;
        if (p < tail) {
            e = lg[p & lmask];
            uint64_t st = 0;
            live = table_find(t, mask, e.key, &st, d.err) >= 0 && st == e.stamp;
        }
        uint32_t tot;
        const uint32_t rk = block_rank(live, s_w, tot);
        if (live) lg[(w + rk) & lmask] = e;   // w + rk <= p: order-preserving, in place
        __syncthreads();
        w += tot;
    }
    if (threadIdx.x == 0) d.log_tail[i] = w;
    if (!rebuild) return;
    __syncthreads();
    for (uint64_t s = threadIdx.x; s < d.S; s += blockDim.x) t[s] = Slot{0, 0};
    __syncthreads();
    for (uint64_t p = front + threadIdx.x; p < w; p += blockDim.x) {
        const Slot e = lg[p & lmask];
        bool claimed = false;
        uint64_t j = e.key & mask;
        for (uint64_t it = 0; it <= mask; ++it) {   // keys are distinct: claim the first empty slot
            const unsigned long long prev =
                atomicCAS(reinterpret_cast<unsigned long long *>(&t[j].key), 0ull, (unsigned long long)e.key);
            if (prev == 0) { t[j].stamp = e.stamp; claimed = true; break; }
            j = (j + 1) & mask;
        }
        if (!claimed) set_err(d.err, DM_ERR_TIMEOUT);
    }
    if (threadIdx.x == 0) d.used[i] = w - front;
}

// Log positions of each request's touches (arrival order per instance), the
// clock base of the batch, and the new log tails.  Single CTA; dynamic smem
// holds one u64 tail per instance.
__global__ void __launch_bounds__(1024) k_commit_prep(DevState d, uint32_t n) {
    extern __shared__ __align__(16) unsigned char smem[];
    if (has_err(d.err)) return;
    uint64_t *tl = reinterpret_cast<uint64_t *>(smem);
    for (uint32_t i = threadIdx.x; i < d.M; i += blockDim.x) tl[i] = d.log_tail[i];
    __syncthreads();
    if (threadIdx.x == 0) {
        for (uint32_t r = 0; r < n; ++r) {
            const uint32_t f = d.r_final[r];
            d.r_touchoff[r] = tl[f];
            tl[f] += d.r_nblk[r];
        }
        d.info->clock_base = *d.clock;
        *d.clock += d.info->total_blocks;
    }
    __syncthreads();
    for (uint32_t i = threadIdx.x; i < d.M; i += blockDim.x) d.log_tail[i] = tl[i];
}

// One warp per 256-block segment: cache keys, stamps, log records, index touches.
__global__ void __launch_bounds__(256) k_commit_touch(DevState d) {
    if (has_err(d.err)) return;
    const int lane = threadIdx.x & 31;
    const uint32_t nwarps = (gridDim.x * blockDim.x) >> 5;
    const uint32_t total_segs = d.info->total_segs;
    const uint64_t clock_base = d.info->clock_base;
    const uint64_t mask = d.S - 1, lmask = d.logcap - 1;
    for (uint32_t seg = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; seg < total_segs; seg += nwarps) {
        const uint32_t r = d.seg_req[seg];
        const uint32_t j = seg - d.r_segoff[r];
        const uint32_t nblk = d.r_nblk[r];
        const uint32_t f = d.r_final[r];
        const uint64_t carry = d.seg_carry[seg];
        const uint64_t bo = d.r_blkoff[r], toff = d.r_touchoff[r];
        Slot *t = d.table[f];
        Slot *lg = d.logbuf[f];
        const uint32_t b_end = min(nblk, (j + 1) * kSegBlocks);
        uint32_t newly = 0, claims = 0;
        for (uint32_t b = j * kSegBlocks + lane; b < b_end; b += 32) {
            const uint64_t key = cache_key(d.plocal[bo + b] + carry, d.Sc);
            const uint64_t stamp = clock_base + bo + (nblk - b);   // block n_blk-1 is touched first
            lg[(toff + (nblk - 1 - b)) & lmask] = Slot{key, stamp};
            bool claimed = false;
            newly += table_touch(t, mask, key, stamp, d.err, &claimed);
            claims += claimed;
        }
        newly = __reduce_add_sync(0xffffffffu, newly);
        claims = __reduce_add_sync(0xffffffffu, claims);
        if (lane == 0) {
            if (newly) atomicAdd(reinterpret_cast<unsigned long long *>(&d.live[f]), (unsigned long long)newly);
            if (claims) atomicAdd(reinterpret_cast<unsigned long long *>(&d.used[f]), (unsigned long long)claims);
        }
    }
}

// Evict the oldest resident keys of every instance above capacity.  CTA per id.
__global__ void __launch_bounds__(1024) k_evict(DevState d) {
    __shared__ uint32_t s_w[33];
    __shared__ uint64_t s_front;
    if (has_err(d.err)) return;
    const uint32_t i = blockIdx.x;
    Slot *t = d.table[i];
    if (!t) return;
    const uint64_t live = d.live[i];
    if (live <= d.C) return;
    Slot *lg = d.logbuf[i];
    const uint64_t mask = d.S - 1, lmask = d.logcap - 1;
    const uint64_t tail = d.log_tail[i];
    uint64_t front = d.log_front[i];
    uint64_t remaining = live - d.C;
    while (remaining > 0 && front < tail) {
        const uint64_t p = front + threadIdx.x;
        int64_t slot = -1;
        bool is_live = false;
        if (p < tail) {
            const Slot e = lg[p & lmask];
            uint64_t st = 0;
            slot = table_find(t, mask, e.key, &st, d.err);
            is_live = slot >= 0 && st == e.stamp;
        }
        uint32_t tot;
        const uint32_t rk = block_rank(is_live, s_w, tot);
        if (threadIdx.x == 0) s_front = min(front + blockDim.x, tail);
        __syncthreads();
        if (is_live && rk < remaining) {
            t[slot].stamp = 0;
            if (rk == remaining - 1) s_front = p + 1;
        }
        __syncthreads();
        front = s_front;
        remaining -= remaining < (uint64_t)tot ? remaining : (uint64_t)tot;
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        if (remaining) set_err(d.err, DM_ERR_TIMEOUT);   // the log must cover every live key
        d.log_front[i] = front;
        d.live[i] = d.C;
    }
}

cudaError_t launch_commit(const DevState &d, uint32_t n, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    cudaError_t e = cudaMemsetAsync(d.touch_cnt, 0, sizeof(uint64_t) * d.M, st);
    if (e != cudaSuccess) return e;
    k_commit_count<<<(n + 255) / 256, 256, 0, st>>>(d, n);
    k_maintain<<<d.M, 1024, 0, st>>>(d);
    const size_t smem = sizeof(uint64_t) * d.M;
    static size_t configured = 0;
    if (smem > configured) {
        e = cudaFuncSetAttribute(k_commit_prep, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        configured = smem;
    }
    k_commit_prep<<<1, 1024, smem, st>>>(d, n);
    k_commit_touch<<<hash_grid_size(), 256, 0, st>>>(d);
    k_evict<<<d.M, 1024, 0, st>>>(d);
    return cudaGetLastError();
}

}  // namespace dm
