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

// Adaptive hash-prefix length (Sec. 3.2): the walk from min(K_route, n_blk)
// blocks, one step deeper while the node (the key of the prefix's last
// block) is expanded.  Level j sits at depth min(d0 + j * step, cap), so
// lane j evaluates level j of each 32-level round at once: the request's
// length is the first level that cannot extend.  Every level passed and the
// final one count toward the window's hotness.  Then the two positions of
// that length.  Whole warp; needs ad_max <= 2048 (segment carries in one
// warp scan).
__device__ __forceinline__ void adaptive_positions(const DevState &d, uint32_t r, int lane, uint64_t &pos1,
                                                   uint64_t &pos2) {
    const uint32_t nblk = d.r_nblk[r], s0 = d.r_segoff[r];
    const uint64_t bo = d.r_blkoff[r];
    const uint32_t d0 = min(d.Kroute, nblk), cap = min(d.ad_max, nblk);
    const uint32_t nseg = (cap - 1) / kSegBlocks + 1;   // <= 32
    const uint64_t t1 = (uint32_t)lane < nseg ? d.seg_total[s0 + lane] : 0;
    const uint64_t t2 = (uint32_t)lane < nseg ? d.seg_total2[s0 + lane] : 0;
    const uint64_t c1 = warp_incl_scan(t1, lane) - t1, c2 = warp_incl_scan(t2, lane) - t2;   // exclusive
    uint32_t K = d0;
    uint64_t P1K = 0;
    for (uint32_t j0 = 0;; j0 += 32) {
        const uint64_t want = uint64_t(d0) + uint64_t(j0 + lane) * d.ad_step;
        const uint32_t dj = want < cap ? (uint32_t)want : cap;
        const uint32_t b = dj - 1;
        const uint64_t P1 = d.plocal[bo + b] + shfl_u64(c1, b / kSegBlocks);
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
    const uint64_t P2K = d.p2local[bo + K - 1] + shfl_u64(c2, (K - 1) / kSegBlocks);
    pos1 = fmix64(P1K ^ d.Sr1);
    pos2 = fmix64(P2K ^ d.Sr2);
    if (lane == 0) d.r_K[r] = K;
}

// One CTA of kProbeWarps warps per request.  Warp 0 computes the two ring
// positions and candidates while warp 1 computes the segment carries; then
// every round probes 32 * kProbeWarps consecutive blocks on each candidate
// still running, and the smallest missing block over the warps ends that
// candidate's run.
constexpr int kProbeWarps = 8;

template <bool kAdapt>
__global__ void __launch_bounds__(kProbeWarps * 32, 4) k_route_probe(DevState d, dm_route_out o, uint32_t n) {
    pdl_enter();
    __shared__ uint32_t s_c[2];
    __shared__ uint32_t s_miss[2][kProbeWarps];
    if (has_err(d.err)) return;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const uint32_t r = blockIdx.x;
    if (wid == 1) {
        request_carries(d, r, lane);   // for the probes below and the commit
    } else if (wid == 0) {
        uint64_t p1, p2;
        if constexpr (kAdapt) {
            adaptive_positions(d, r, lane, p1, p2);
        } else {
            route_positions_direct(d, r, lane, p1, p2);
            if (lane == 0) d.r_K[r] = min(d.Kroute, d.r_nblk[r]);
        }
        uint32_t lb1, lb2;
        ring_search2(d, p1, p2, lane, lb1, lb2);
        const uint32_t c1 = d.ring[0].owner[lb1];
        const uint32_t raw2 = d.ring[1].owner[lb2];
        if (lane == 0) {
            s_c[0] = c1;
            s_c[1] = raw2 != c1 ? raw2 : d.next_live[c1];
        }
    }
    __syncthreads();
    const uint32_t c1 = s_c[0], c2 = s_c[1];
    const uint32_t nblk = d.r_nblk[r], s0 = d.r_segoff[r];
    const uint64_t bo = d.r_blkoff[r];
    const Slot *t1 = d.table[c1];
    const Slot *t2 = d.table[c2];
    const uint64_t f1 = d.log_front[c1], f2 = d.log_front[c2];   // resident: record at or after the front
    const uint64_t mask = d.S - 1;
    constexpr uint32_t kRound = 32 * kProbeWarps;
    bool done1 = false, done2 = false;
    uint32_t h1 = 0, h2 = 0;
    for (uint32_t base = 0; !(done1 && done2); base += kRound) {
        const uint32_t b = base + threadIdx.x;   // base is a multiple of the group size
        const bool inb = b < nblk;
        bool res1 = false, res2 = false;
        const uint64_t key = inb ? cache_key(d.plocal[bo + b] + d.seg_carry[s0 + b / kSegBlocks], d.Sc) : 0;
        const uint64_t home = group_home(group_anchor(key, lane), b, mask);
        if (inb) {
            if (!done1) res1 = table_pos1(t1, mask, key, home, d.err) > f1;
            if (!done2) res2 = table_pos1(t2, mask, key, home, d.err) > f2;
        }
        const uint32_t m1 = __ballot_sync(0xffffffffu, !res1);
        const uint32_t m2 = __ballot_sync(0xffffffffu, !res2);
        if (lane == 0) {
            s_miss[0][wid] = m1 ? wid * 32 + __ffs(m1) - 1 : kRound;
            s_miss[1][wid] = m2 ? wid * 32 + __ffs(m2) - 1 : kRound;
        }
        __syncthreads();
        uint32_t m1w = kRound, m2w = kRound;
#pragma unroll
        for (int w = 0; w < kProbeWarps; ++w) {
            m1w = min(m1w, s_miss[0][w]);
            m2w = min(m2w, s_miss[1][w]);
        }
        if (!done1 && m1w < kRound) { h1 = base + m1w; done1 = true; }
        if (!done2 && m2w < kRound) { h2 = base + m2w; done2 = true; }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
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
    if (d.ad_step)
        DM_TRY(launch_pdl(k_route_probe<true>, b.n, kProbeWarps * 32, 0, st, d, o, b.n));
    else
        DM_TRY(launch_pdl(k_route_probe<false>, b.n, kProbeWarps * 32, 0, st, d, o, b.n));
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

namespace dm {

// End of an adaptive window: new_set (cleared) receives the expanded nodes
// that stay (reached by at least T/n requests) and the nodes that become
// expanded (reached by more than 2T/n, shorter than the cap).  Grid-stride
// over both tables.
__global__ void k_adapt_update(DevState d, uint64_t *new_set, uint64_t n_live, uint64_t T) {
    pdl_enter();
    if (has_err(d.err)) return;
    const uint64_t ns = d.ad_set_mask + 1, nc = d.ad_cnt_mask + 1, tot = ns > nc ? ns : nc;
    const uint64_t stride = uint64_t(gridDim.x) * blockDim.x;
    for (uint64_t x = uint64_t(blockIdx.x) * blockDim.x + threadIdx.x; x < tot; x += stride) {
        if (x < ns) {
            const uint64_t key = d.ad_set[x];
            if (key) {
                const uint64_t c = ad_count_get(d.ad_cnt, d.ad_cnt_mask, key, d.err);
                if (!(c * n_live < T)) ad_set_insert(new_set, d.ad_set_mask, key, d.err);
            }
        }
        if (x < nc) {
            const AdCount e = d.ad_cnt[x];
            if (e.key && e.depth < d.ad_max && uint64_t(e.count) * n_live > 2 * T &&
                !ad_set_contains(d.ad_set, d.ad_set_mask, e.key, d.err))
                ad_set_insert(new_set, d.ad_set_mask, e.key, d.err);
        }
    }
}

cudaError_t launch_adapt_update(const DevState &d, uint64_t *new_set, uint64_t n_live, uint64_t T, cudaStream_t st) {
    const uint64_t tot = (d.ad_set_mask > d.ad_cnt_mask ? d.ad_set_mask : d.ad_cnt_mask) + 1;
    const unsigned grid = (unsigned)((tot + 255) / 256 < 4096 ? (tot + 255) / 256 : 4096);
    DM_TRY(launch_pdl(k_adapt_update, grid, 256, 0, st, d, new_set, n_live, T));
    return cudaGetLastError();
}

}  // namespace dm
