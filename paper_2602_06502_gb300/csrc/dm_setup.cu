// dm_setup.cu -- batch set-up: validation of the prompts, per-request block
// and segment offsets (and, for routing, the offsets of the hashing order),
// the segment -> request map of the hashing-only calls, and (in the same
// launch as the set-up, routing calls only) the queue drain of Sec. 3.2.
#include "dm_internal.cuh"

namespace dm {

// ---------------------------------------------------------------------------
// Block-wide exclusive scan of three 64-bit counters (1024 threads).
__device__ __forceinline__ void block_scan3(const uint64_t (&v)[3], uint64_t (&ex)[3], uint64_t (&tot)[3],
                                            uint64_t (*sm)[32]) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    uint64_t inc[3];
#pragma unroll
    for (int k = 0; k < 3; ++k) {
        inc[k] = warp_incl_scan(v[k], lane);
        if (lane == 31) sm[k][wid] = inc[k];
    }
    __syncthreads();
    if (wid == 0) {
#pragma unroll
        for (int k = 0; k < 3; ++k) sm[k][lane] = warp_incl_scan(sm[k][lane], lane);   // inclusive over warps
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < 3; ++k) {
        ex[k] = (wid ? sm[k][wid - 1] : 0) + inc[k] - v[k];
        tot[k] = sm[k][31];
    }
    __syncthreads();
}

// CTA 0: validate the batch and lay out per-request block / segment
// offsets.  Routing only (kRoute): the offsets of the routing kernel's task
// order (routing columns, rest of the head below d.H, tail), both
// candidates' first-miss slots set to "none", and the routing kernel's list
// counters; CTA 1 folds the previous batch's pending CV sample into the
// metrics; CTAs 2.. drain the queues by `delta` us from time t0 on, a warp
// per instance (independent of the batch layout).
template <bool kRoute>
__global__ void __launch_bounds__(1024) k_setup(DevState d, const uint64_t *off, const uint32_t *len,
                                                uint32_t n, uint64_t total_tokens, uint64_t delta, uint64_t t0) {
    pdl_enter();
    __shared__ uint64_t sm[3][32];
    if (has_err(d.err)) return;
    if (blockIdx.x == 1) {   // the previous batch's CV sample (beside the layout)
        if (threadIdx.x == 0) fold_cv(d.metrics);
        return;
    }
    if (blockIdx.x > 1) {
        const uint32_t i = (blockIdx.x - 2) * (blockDim.x >> 5) + (threadIdx.x >> 5);
        if (i < d.M) drain_queue(d, i, delta, t0, threadIdx.x & 31);
        return;
    }
    // [0] blocks; [1] kRoute: head segments past the routing columns | (segments
    // in the routing columns) << 32, else segments; [2] kRoute: tail segments
    uint64_t carry[3] = {0, 0, 0};
    bool bad = false;
    for (uint32_t base = 0; base < n; base += blockDim.x) {
        uint32_t r = base + threadIdx.x;
        uint64_t nblk = 0;
        uint32_t nseg = 0;
        if (r < n) {
            uint32_t L = len[r];
            uint64_t o = off[r];
            if (L < d.B || (o & 3) || o > total_tokens || L > total_tokens - o) {
                bad = true;
            } else {
                nblk = L / d.B;
                nseg = (uint32_t)((nblk + kSegBlocks - 1) / kSegBlocks);
            }
            d.r_L[r] = L;
            d.r_nblk[r] = (uint32_t)nblk;
            d.r_tokoff[r] = o;
        }
        const uint32_t hs = min(nseg, d.H), cs = min(nseg, d.Ccols);
        const uint64_t v[3] = {nblk, kRoute ? (uint64_t(cs) << 32 | (hs - cs)) : nseg,
                               kRoute ? uint64_t(nseg - hs) : 0};
        uint64_t ex[3], tot[3];
        block_scan3(v, ex, tot, sm);
        if (r < n) {
            d.r_blkoff[r] = carry[0] + ex[0];
            if constexpr (kRoute) {
                const uint64_t e1 = carry[1] + ex[1];
                const uint32_t ho = (uint32_t)e1, co = (uint32_t)(e1 >> 32), to = (uint32_t)(carry[2] + ex[2]);
                d.r_hoff[r] = ho;
                d.r_toff[r] = to;
                d.r_segoff[r] = co + ho + to;
            } else {
                d.r_segoff[r] = (uint32_t)(carry[1] + ex[1]);
            }
        }
#pragma unroll
        for (int k = 0; k < 3; ++k) carry[k] += tot[k];
    }
    if (bad) set_err(d.err, DM_ERR_INVALID_ARG);
    if (threadIdx.x == 0) {
        const uint64_t hr = carry[1] & 0xFFFFFFFFull, cols = carry[1] >> 32;
        const uint64_t segs = kRoute ? hr + cols + carry[2] : carry[1];
        d.info->total_blocks = carry[0];
        d.info->total_segs = (uint32_t)segs;
        d.info->head_segs = kRoute ? (uint32_t)hr : 0u;
        d.info->col_tasks = kRoute ? n * d.Ccols : 0u;
        d.info->tasks = kRoute ? (uint32_t)(uint64_t(n) * d.Ccols + hr + carry[2]) : 0u;
        d.info->n = n;
        d.info->both_over = 0;
        d.info->fix_n = 0;
        d.info->cta_done = 0;
        if (carry[0] > d.max_blocks || segs > d.max_segs || uint64_t(n) * d.Ccols + segs >= (1ull << 32))
            set_err(d.err, DM_ERR_CAPACITY);
    }
}

// Segment -> request map, one warp per request.
__global__ void k_segmap(DevState d, uint32_t n) {
    pdl_enter();
    if (has_err(d.err)) return;
    const int lane = threadIdx.x & 31;
    const uint32_t r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (r >= n) return;
    const uint32_t s0 = d.r_segoff[r];
    const uint32_t ns = (d.r_nblk[r] + kSegBlocks - 1) / kSegBlocks;
    for (uint32_t j = lane; j < ns; j += 32) d.seg_req[s0 + j] = r;
}

cudaError_t launch_setup(const DevState &d, const dm_batch &b, cudaStream_t st) {
    DM_TRY(launch_pdl(k_setup<false>, 1, 1024, 0, st, d, b.offsets, b.lengths, b.n, b.total_tokens, uint64_t(0),
                      uint64_t(0)));
    if (b.n) DM_TRY(launch_pdl(k_segmap, (b.n + 7) / 8, 256, 0, st, d, b.n));
    return cudaGetLastError();
}

// Routing with d candidates: the plain layout (segment order, then the
// segment -> request map), the CV fold and the queue drain.
cudaError_t launch_setup_plain_drain(const DevState &d, const dm_batch &b, uint64_t delta, uint64_t t0,
                                     cudaStream_t st) {
    const unsigned drain_ctas = (d.M + 31) / 32;
    DM_TRY(launch_pdl(k_setup<false>, 2 + drain_ctas, 1024, 0, st, d, b.offsets, b.lengths, b.n, b.total_tokens,
                      delta, t0));
    if (b.n) DM_TRY(launch_pdl(k_segmap, (b.n + 7) / 8, 256, 0, st, d, b.n));
    return cudaGetLastError();
}

// Routing: the layout in the hashing order of k_hash_probe (which writes
// the segment -> request map itself), the CV fold and the queue drain.
cudaError_t launch_setup_route(const DevState &d, const dm_batch &b, uint64_t delta, uint64_t t0,
                               cudaStream_t st) {
    const unsigned drain_ctas = (d.M + 31) / 32;
    DM_TRY(launch_pdl(k_setup<true>, 2 + drain_ctas, 1024, 0, st, d, b.offsets, b.lengths, b.n, b.total_tokens,
                      delta, t0));
    return cudaGetLastError();
}

}  // namespace dm
