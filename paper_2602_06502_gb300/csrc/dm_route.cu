// dm_route.cu -- dual-ring lookup, distinct-candidate fix and cache probes
// (Sec. 3.2, Sec. 3.4, App. A.1.3, App. A.3.2).
//
// Ring search: each ring is a sorted array of virtual-node positions plus a
// static 32-ary search tree (level k holds every 32^k-th position).  A warp
// compares one 256-byte row of 32 keys per level and ballots, so a ring of
// 262,144 nodes takes four coalesced L2 reads.  The successor of p is the
// first node with position >= p, wrapping to node 0.
//
// Probes: lane l tests block 32*it + l of the prompt against a candidate's
// open-addressed index; the first zero bit of the warp ballot ends the
// leading run of resident keys.
#include "dm_internal.cuh"

namespace dm {

__device__ __forceinline__ const uint64_t *level_ptr(const DevState &d, int f, int k) {
    return k == 0 ? d.ring[f].vpos : d.ring[f].tree + d.lev_off[k];
}

// Index (level 0) of the successor of p1 on ring 0 and of p2 on ring 1.
// Whole warp; the two searches are interleaved for memory-level parallelism.
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

// One warp per request: carries, candidates, hit lengths.
__global__ void __launch_bounds__(128) k_route_probe(DevState d, dm_route_out o, uint32_t n) {
    if (has_err(d.err)) return;
    const int lane = threadIdx.x & 31;
    const uint32_t r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (r >= n) return;
    request_carries(d, r, lane);
    __syncwarp();

    uint32_t lb1, lb2;
    ring_search2(d, d.r_pos[2 * r], d.r_pos[2 * r + 1], lane, lb1, lb2);
    const uint32_t c1 = d.ring[0].owner[lb1];
    const uint32_t raw2 = d.ring[1].owner[lb2];
    const uint32_t c2 = raw2 != c1 ? raw2 : d.next_live[c1];

    const uint32_t nblk = d.r_nblk[r], s0 = d.r_segoff[r];
    const uint64_t bo = d.r_blkoff[r];
    const Slot *t1 = d.table[c1];
    const Slot *t2 = d.table[c2];
    const uint64_t mask = d.S - 1;
    bool done1 = false, done2 = false;
    uint32_t h1 = 0, h2 = 0;
    for (uint32_t it = 0; !(done1 && done2); ++it) {
        const uint32_t b = it * 32 + lane;
        const bool inb = b < nblk;
        bool res1 = false, res2 = false;
        if (inb) {
            const uint64_t key = cache_key(d.plocal[bo + b] + d.seg_carry[s0 + b / kSegBlocks], d.Sc);
            uint64_t st;
            if (!done1) res1 = table_find(t1, mask, key, &st, d.err) >= 0 && st != 0;
            if (!done2) res2 = table_find(t2, mask, key, &st, d.err) >= 0 && st != 0;
        }
        const uint32_t m1 = __ballot_sync(0xffffffffu, !res1);
        const uint32_t m2 = __ballot_sync(0xffffffffu, !res2);
        if (!done1 && m1) { h1 = it * 32 + __ffs(m1) - 1; done1 = true; }
        if (!done2 && m2) { h2 = it * 32 + __ffs(m2) - 1; done2 = true; }
    }
    if (lane == 0) {
        const uint32_t hit1 = h1 * d.B, hit2 = h2 * d.B;
        d.r_c1[r] = c1;
        d.r_c2[r] = c2;
        d.r_h1[r] = hit1;
        d.r_h2[r] = hit2;
        o.cand1[r] = c1;
        o.cand2[r] = c2;
        o.hit1[r] = hit1;
        o.hit2[r] = hit2;
    }
}

cudaError_t launch_route_probe(const DevState &d, const dm_batch &b, const dm_route_out &o,
                               cudaStream_t st) {
    if (b.n == 0) return cudaSuccess;
    const uint32_t warps = 4;
    k_route_probe<<<(b.n + warps - 1) / warps, warps * 32, 0, st>>>(d, o, b.n);
    return cudaGetLastError();
}

// dm_ring_lookup: raw owners of (pos1, pos2) pairs, one warp per pair.
__global__ void k_ring_lookup(DevState d, const uint64_t *pos, uint32_t n, uint32_t *o1, uint32_t *o2) {
    if (has_err(d.err)) return;
    const int lane = threadIdx.x & 31;
    const uint32_t r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (r >= n) return;
    uint32_t lb1, lb2;
    ring_search2(d, pos[2 * r], pos[2 * r + 1], lane, lb1, lb2);
    if (lane == 0) {
        o1[r] = d.ring[0].owner[lb1];
        o2[r] = d.ring[1].owner[lb2];
    }
}

cudaError_t launch_ring_lookup(const DevState &d, const uint64_t *pos, uint32_t n, uint32_t *o1,
                               uint32_t *o2, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    k_ring_lookup<<<(n + 7) / 8, 256, 0, st>>>(d, pos, n, o1, o2);
    return cudaGetLastError();
}

}  // namespace dm
