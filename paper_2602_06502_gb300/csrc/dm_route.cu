// dm_route.cu -- standalone dual-ring lookup (dm_ring_lookup; Sec. 3.2,
// Sec. 3.4, App. A.1.3) and the end-of-window update of the adaptive
// prefix tree (Sec. 3.2).  The routing kernel itself (hashing, ring
// lookup, distinct fix and probes in one pass) is in dm_hash.cu.
#include "dm_internal.cuh"

namespace dm {

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
