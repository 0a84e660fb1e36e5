// dm_setup.cu -- batch set-up: validation of the prompts, per-request block
// and segment offsets, the segment -> request map, and (in the same launch
// as the set-up, routing calls only) the queue drain of Sec. 3.2.
#include "dm_internal.cuh"

namespace dm {

// ---------------------------------------------------------------------------
// Block-wide exclusive scan of two counters (1024 threads).
__device__ __forceinline__ void block_scan2(uint64_t a, uint32_t b, uint64_t &ea, uint32_t &eb,
                                            uint64_t &ta, uint32_t &tb, uint64_t *sa, uint32_t *sb) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    uint64_t ia = a;
    uint32_t ib = b;
#pragma unroll
    for (int dd = 1; dd < 32; dd <<= 1) {
        uint64_t ua = __shfl_up_sync(0xffffffffu, ia, dd);
        uint32_t ub = __shfl_up_sync(0xffffffffu, ib, dd);
        if (lane >= dd) { ia += ua; ib += ub; }
    }
    if (lane == 31) { sa[wid] = ia; sb[wid] = ib; }
    __syncthreads();
    if (wid == 0) {
        uint64_t wa = sa[lane];
        uint32_t wb = sb[lane];
#pragma unroll
        for (int dd = 1; dd < 32; dd <<= 1) {
            uint64_t ua = __shfl_up_sync(0xffffffffu, wa, dd);
            uint32_t ub = __shfl_up_sync(0xffffffffu, wb, dd);
            if (lane >= dd) { wa += ua; wb += ub; }
        }
        sa[lane] = wa;   // inclusive over warps
        sb[lane] = wb;
    }
    __syncthreads();
    uint64_t pa = wid ? sa[wid - 1] : 0;
    uint32_t pb = wid ? sb[wid - 1] : 0;
    ea = pa + ia - a;
    eb = pb + ib - b;
    ta = sa[31];
    tb = sb[31];
    __syncthreads();
}

// CTA 0: validate the batch and lay out per-request block / segment
// offsets.  Routing only: CTA 1 folds the previous batch's pending CV
// sample into the metrics; CTAs 2.. drain the queues by `delta` us from
// time t0 on, a warp per instance (independent of the batch layout).
__global__ void __launch_bounds__(1024) k_setup(DevState d, const uint64_t *off, const uint32_t *len,
                                                uint32_t n, uint64_t total_tokens, uint64_t delta, uint64_t t0) {
    pdl_enter();
    __shared__ uint64_t sa[32];
    __shared__ uint32_t sb[32];
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
    uint64_t carry_blk = 0;
    uint32_t carry_seg = 0;
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
        uint64_t eblk, tblk;
        uint32_t eseg, tseg;
        block_scan2(nblk, nseg, eblk, eseg, tblk, tseg, sa, sb);
        if (r < n) {
            d.r_blkoff[r] = carry_blk + eblk;
            d.r_segoff[r] = carry_seg + eseg;
        }
        carry_blk += tblk;
        carry_seg += tseg;
    }
    if (bad) set_err(d.err, DM_ERR_INVALID_ARG);
    if (threadIdx.x == 0) {
        d.info->total_blocks = carry_blk;
        d.info->total_segs = carry_seg;
        d.info->n = n;
        d.info->both_over = 0;
        if (carry_blk > d.max_blocks || carry_seg > d.max_segs) set_err(d.err, DM_ERR_CAPACITY);
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
    DM_TRY(launch_pdl(k_setup, 1, 1024, 0, st, d, b.offsets, b.lengths, b.n, b.total_tokens, uint64_t(0),
                      uint64_t(0)));
    if (b.n) DM_TRY(launch_pdl(k_segmap, (b.n + 7) / 8, 256, 0, st, d, b.n));
    return cudaGetLastError();
}

cudaError_t launch_setup_drain(const DevState &d, const dm_batch &b, uint64_t delta, uint64_t t0,
                               cudaStream_t st) {
    const unsigned drain_ctas = (d.M + 31) / 32;
    DM_TRY(launch_pdl(k_setup, 2 + drain_ctas, 1024, 0, st, d, b.offsets, b.lengths, b.n, b.total_tokens, delta,
                      t0));
    if (b.n) DM_TRY(launch_pdl(k_segmap, (b.n + 7) / 8, 256, 0, st, d, b.n));
    return cudaGetLastError();
}

}  // namespace dm
