// dm_ring.cu -- dual consistent-hash rings with virtual nodes (Sec. 3.4,
// App. A.1.3; d rings for the d-candidate path of App. A.8).  Each live id
// owns V nodes per ring at
//   vpos_f(id, v) = fmix64(splitmix_step((id << 32) | v) ^ S_vf),
// kept sorted by (position, id, v).  Adding an id inserts its V nodes,
// removing it deletes them; all other nodes keep their relative order, so
// only keys on the changed arcs remap.
//
// Both updates rank in parallel: the id's V nodes are generated and sorted
// (one CTA, bitonic), then every surviving old node moves by the number of
// id nodes before it and every new node lands at (its rank among the new
// nodes + number of old nodes before it), found by binary search.
#include "dm_internal.cuh"

namespace dm {

struct VNode {
    uint64_t pos;
    uint32_t id, v;
};

__device__ __forceinline__ bool vless(uint64_t pa, uint32_t ia, uint32_t va, uint64_t pb, uint32_t ib,
                                      uint32_t vb) {
    if (pa != pb) return pa < pb;
    if (ia != ib) return ia < ib;
    return va < vb;
}

// Vnode seed of ring f.
__device__ __forceinline__ uint64_t ring_seed(const DevState &d, int f) {
    return f == 0 ? d.Sv1 : f == 1 ? d.Sv2 : d.Svx[f - 2];
}

// Generate and sort the V nodes of `id` for every ring (one CTA per ring).
__global__ void __launch_bounds__(1024) k_gen_sort(DevState d, uint32_t id, uint64_t *spos, uint32_t *svidx,
                                                   uint32_t P) {
    const int f = blockIdx.x;
    const uint64_t Sv = ring_seed(d, f);
    uint64_t *pos = spos + uint64_t(f) * P;
    uint32_t *vi = svidx + uint64_t(f) * P;
    for (uint32_t v = threadIdx.x; v < P; v += blockDim.x) {
        pos[v] = v < d.V ? vnode_pos(Sv, id, v) : ~0ull;
        vi[v] = v < d.V ? v : 0xFFFFFFFFu;
    }
    __syncthreads();
    for (uint32_t k = 2; k <= P; k <<= 1) {
        for (uint32_t j = k >> 1; j > 0; j >>= 1) {
            for (uint32_t x = threadIdx.x; x < P; x += blockDim.x) {
                const uint32_t y = x ^ j;
                if (y > x) {
                    const bool asc = (x & k) == 0;
                    const bool gt = vless(pos[y], id, vi[y], pos[x], id, vi[x]);  // x > y
                    if (gt == asc) {
                        const uint64_t tp = pos[x]; pos[x] = pos[y]; pos[y] = tp;
                        const uint32_t tv = vi[x]; vi[x] = vi[y]; vi[y] = tv;
                    }
                }
            }
            __syncthreads();
        }
    }
}

// Number of entries of the sorted id-node list (all owned by `id`) that
// precede (p, o, v).
__device__ __forceinline__ uint32_t count_new_before(const uint64_t *npos, const uint32_t *nvi, uint32_t V,
                                                     uint32_t id, uint64_t p, uint32_t o, uint32_t v) {
    uint32_t lo = 0, hi = V;
    while (lo < hi) {
        const uint32_t mid = (lo + hi) >> 1;
        if (vless(npos[mid], id, nvi[mid], p, o, v)) lo = mid + 1; else hi = mid;
    }
    return lo;
}

// Destination buffers of every ring.
struct RingSet {
    Ring r[kMaxD];
};

// Add: old nodes shift right, new nodes are placed; every ring (blockIdx.y).
__global__ void k_merge_add(DevState d, uint32_t id, const uint64_t *spos, const uint32_t *svidx, uint32_t P,
                            RingSet dsts) {
    const int f = blockIdx.y;
    const Ring src = d.ring[f];
    const Ring dst = dsts.r[f];
    const uint64_t *npos = spos + uint64_t(f) * P;
    const uint32_t *nvi = svidx + uint64_t(f) * P;
    const uint32_t R = d.R, V = d.V;
    const uint32_t t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t < R) {
        const uint64_t p = src.vpos[t];
        const uint32_t o = src.owner[t], v = src.vidx[t];
        const uint32_t k = t + count_new_before(npos, nvi, V, id, p, o, v);
        dst.vpos[k] = p;
        dst.owner[k] = o;
        dst.vidx[k] = v;
    } else if (t < R + V) {
        const uint32_t j = t - R;
        const uint64_t p = npos[j];
        const uint32_t v = nvi[j];
        uint32_t lo = 0, hi = R;   // old nodes before (p, id, v)
        while (lo < hi) {
            const uint32_t mid = (lo + hi) >> 1;
            if (vless(src.vpos[mid], src.owner[mid], src.vidx[mid], p, id, v)) lo = mid + 1; else hi = mid;
        }
        const uint32_t k = j + lo;
        dst.vpos[k] = p;
        dst.owner[k] = id;
        dst.vidx[k] = v;
    }
}

// Remove: surviving nodes shift left by the id nodes that precede them.
__global__ void k_merge_remove(DevState d, uint32_t id, const uint64_t *spos, const uint32_t *svidx, uint32_t P,
                               RingSet dsts) {
    const int f = blockIdx.y;
    const Ring src = d.ring[f];
    const Ring dst = dsts.r[f];
    const uint64_t *npos = spos + uint64_t(f) * P;
    const uint32_t *nvi = svidx + uint64_t(f) * P;
    const uint32_t t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= d.R) return;
    const uint32_t o = src.owner[t];
    if (o == id) return;
    const uint64_t p = src.vpos[t];
    const uint32_t v = src.vidx[t];
    const uint32_t k = t - count_new_before(npos, nvi, d.V, id, p, o, v);
    dst.vpos[k] = p;
    dst.owner[k] = o;
    dst.vidx[k] = v;
}

cudaError_t launch_ring_update(DevState &d, uint32_t id, bool add, uint64_t *scratch_pos, uint32_t *scratch_vidx,
                               uint64_t *const *new_vpos, uint32_t *const *new_owner, uint32_t *const *new_vidx,
                               cudaStream_t st) {
    uint32_t P = 1;
    while (P < d.V) P <<= 1;
    k_gen_sort<<<d.nrings, 1024, 0, st>>>(d, id, scratch_pos, scratch_vidx, P);
    RingSet dst{};
    for (uint32_t f = 0; f < d.nrings; ++f) {
        dst.r[f].vpos = new_vpos[f];
        dst.r[f].owner = new_owner[f];
        dst.r[f].vidx = new_vidx[f];
        dst.r[f].tree = d.ring[f].tree;
    }
    const uint32_t work = add ? d.R + d.V : d.R;
    if (work > 0) {
        dim3 grid((work + 255) / 256, d.nrings);
        if (add)
            k_merge_add<<<grid, 256, 0, st>>>(d, id, scratch_pos, scratch_vidx, P, dst);
        else
            k_merge_remove<<<grid, 256, 0, st>>>(d, id, scratch_pos, scratch_vidx, P, dst);
    }
    return cudaGetLastError();
}

// Search-tree levels k >= 1: level k entry i = vpos[i * 32^k].
__global__ void k_tree(DevState d) {
    const int f = blockIdx.y;
    const uint64_t t = uint64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    uint64_t stride = 32;
    for (uint32_t k = 1; k < d.nlev; ++k, stride *= 32) {
        if (t < d.lev_n[k]) d.ring[f].tree[d.lev_off[k] + t] = d.ring[f].vpos[t * stride];
    }
}

cudaError_t launch_tree_build(const DevState &d, cudaStream_t st) {
    if (d.nlev <= 1) return cudaSuccess;
    dim3 grid((uint32_t)((d.lev_n[1] + 255) / 256), d.nrings);
    k_tree<<<grid, 256, 0, st>>>(d);
    return cudaGetLastError();
}

// next_live[i] = the next live id after i in ascending order, cyclically.
__global__ void k_next_live(DevState d) {
    const uint32_t i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= d.M) return;
    uint32_t nx = i;
    for (uint32_t k = 1; k <= d.M; ++k) {
        const uint32_t j = (i + k) % d.M;
        if (d.inst_state[j] == 1) { nx = j; break; }
    }
    d.next_live[i] = nx;
}

cudaError_t launch_next_live(const DevState &d, cudaStream_t st) {
    k_next_live<<<(d.M + 255) / 256, 256, 0, st>>>(d);
    return cudaGetLastError();
}

}  // namespace dm

namespace dm {

__global__ void k_set_state(DevState d, uint32_t id, uint8_t s) { d.inst_state[id] = s; }

cudaError_t launch_set_state(const DevState &d, uint32_t id, uint8_t s, cudaStream_t st) {
    k_set_state<<<1, 1, 0, st>>>(d, id, s);
    return cudaGetLastError();
}

}  // namespace dm
