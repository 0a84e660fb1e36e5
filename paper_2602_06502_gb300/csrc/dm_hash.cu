// dm_hash.cu -- prompt hashing (Sec. 3.2: two independent hash functions
// over the prompt prefix; App. A.1.1 block-granular keys).  The batch layout
// it reads is made by dm_setup.cu.
//
// Per full block k of a prompt (B tokens t_0..t_{B-1}) under function f:
//   nh^f_k = sum_i ((t_2i + K^f_2i) mod 2^32) * ((t_2i+1 + K^f_2i+1) mod 2^32)  mod 2^64
//   d^f_k  = fmix64(nh^f_k + (k+1) G^f)
//   P^f_b  = sum_{k<=b} d^f_k  mod 2^64
// Because the chain is a plain prefix sum, every 64-block segment of every
// prompt is hashed independently (one warp each); a segment writes its local
// prefix values and its totals, and the probe kernel adds the carry of the
// earlier segments.  f2 only runs over the first K = min(Kf2, n_blk) blocks
// (Kf2 = K_route, or the longest adaptive prefix): segments below K write the
// sum of their f2 digests and, with the adaptive length, each block's
// in-segment f2 prefix value.
#include "dm_internal.cuh"

namespace dm {

// ---------------------------------------------------------------------------
// Streaming 16-byte load: read once, do not keep in L1.
__device__ __forceinline__ uint4 ld_stream(const uint4 *p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(__cvta_generic_to_global(p)));
    return v;
}

// NH partial over 4 consecutive tokens (two pairs) with the lane's 4 keys.
__device__ __forceinline__ uint64_t nh4(uint4 t, const uint32_t (&k)[4]) {
    return uint64_t(t.x + k[0]) * uint64_t(t.y + k[1]) + uint64_t(t.z + k[2]) * uint64_t(t.w + k[3]);
}

// Within each group of U lanes, lane q holds U partial sums (one per load
// j); after log2(U) exchange steps lane q holds the full sum for j == q.
template <int U>
__device__ __forceinline__ uint64_t reduce_scatter(uint64_t (&p)[U], int q) {
#pragma unroll
    for (int s = U / 2; s >= 1; s >>= 1) {
        const bool hi = (q & s) != 0;
#pragma unroll
        for (int j = 0; j < s; ++j) {
            uint64_t lo_v = p[j], hi_v = p[j + s];
            uint64_t send = hi ? lo_v : hi_v;
            uint64_t keep = hi ? hi_v : lo_v;
            p[j] = keep + shfl_xor_u64(send, s);
        }
    }
    return p[0];
}

// One warp per segment of up to 64 blocks (two iterations of 32 blocks).
// Iteration `it` covers 32 blocks (32*U uint4): load j of lane l reads uint4
// j*32+l of the iteration (fully coalesced), which is quarter l%U of block
// j*(32/U)+l/U.  Both iterations' loads are issued before any arithmetic
// (4 KB in flight per warp at B = 16).  After the reduce-scatter lane l
// holds block (l%U)*(32/U) + l/U; one shuffle puts block m on lane m for the
// scan.  Segments below K also sum their f2 digests (blocks < K); kP2 adds
// their per-block prefix values (the adaptive length picks its K later).
template <int U, bool kP2>
__global__ void __launch_bounds__(256, 4) k_hash(DevState d, const uint32_t *__restrict__ tokens) {
    pdl_enter();
    constexpr int IT = kSegBlocks / 32;
    if (has_err(d.err)) return;
    const int lane = threadIdx.x & 31;
    const uint32_t nwarps = (gridDim.x * blockDim.x) >> 5;
    const uint32_t gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint32_t total_segs = d.info->total_segs;
    constexpr int GPL = 32 / U;  // blocks per load instruction
    const int q = lane % U, g = lane / U;
    const int bq = q * GPL + g;                    // block this lane reduces
    const int src = (lane % GPL) * U + lane / GPL; // lane holding block `lane`
    uint32_t k1[4], k2[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) { k1[i] = d.K1[4 * q + i]; k2[i] = d.K2[4 * q + i]; }
    const uint64_t G1 = d.G1, G2 = d.G2;

    for (uint32_t seg = gw; seg < total_segs; seg += nwarps) {
        const uint32_t r = d.seg_req[seg];
        const uint32_t j = seg - d.r_segoff[r];
        const uint32_t nblk = d.r_nblk[r];
        const uint32_t b0 = j * kSegBlocks;
        const uint32_t nb = min(kSegBlocks, nblk - b0);
        const uint4 *src4 = reinterpret_cast<const uint4 *>(tokens + d.r_tokoff[r] + uint64_t(b0) * d.B);
        uint64_t *out = d.plocal + d.r_blkoff[r] + b0;
        const uint32_t K = min(d.Kf2, nblk);
        uint4 v[IT][U];
#pragma unroll
        for (int it = 0; it < IT; ++it)
#pragma unroll
            for (int jj = 0; jj < U; ++jj) {
                const uint32_t blk = it * 32 + jj * GPL + g;
                v[it][jj] = blk < nb ? ld_stream(src4 + uint64_t(it) * 32 * U + jj * 32 + lane)
                                     : make_uint4(0, 0, 0, 0);
            }
        uint64_t carry1 = 0, sum2 = 0;   // kP2: sum2 is the running f2 prefix (uniform)
#pragma unroll
        for (int it = 0; it < IT; ++it) {
            if ((uint32_t)it * 32 >= nb) break;
            const uint32_t nvalid = min(32u, nb - it * 32);
            uint64_t p1[U];
#pragma unroll
            for (int jj = 0; jj < U; ++jj) p1[jj] = nh4(v[it][jj], k1);
            const uint64_t s1 = reduce_scatter<U>(p1, q);
            const uint32_t kb = b0 + it * 32 + bq;   // block index within the prompt
            uint64_t dg1 = (uint32_t)bq < nvalid ? fmix64(s1 + uint64_t(kb + 1) * G1) : 0;
            dg1 = shfl_u64(dg1, src);
            const uint64_t P1 = warp_incl_scan(dg1, lane) + carry1;
            if ((uint32_t)lane < nvalid) out[it * 32 + lane] = P1;
            carry1 = shfl_u64(P1, 31);
            if (b0 + it * 32 < K) {                   // second function, blocks < K
                uint64_t p2[U];
#pragma unroll
                for (int jj = 0; jj < U; ++jj) p2[jj] = nh4(v[it][jj], k2);
                const uint64_t s2 = reduce_scatter<U>(p2, q);
                const uint64_t dg2 = ((uint32_t)bq < nvalid && kb < K) ? fmix64(s2 + uint64_t(kb + 1) * G2) : 0;
                if constexpr (kP2) {
                    const uint64_t P2 = warp_incl_scan(shfl_u64(dg2, src), lane) + sum2;
                    if ((uint32_t)lane < nvalid && b0 + it * 32 + lane < K)
                        d.p2local[d.r_blkoff[r] + b0 + it * 32 + lane] = P2;
                    sum2 = shfl_u64(P2, 31);
                } else {
                    sum2 += dg2;
                }
            }
        }
        if constexpr (!kP2) {
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1) sum2 += shfl_xor_u64(sum2, o);
        }
        if (lane == 0) {
            d.seg_total[seg] = carry1;
            d.seg_total2[seg] = sum2;
        }
    }
}

int hash_grid_size() {
    static int grid = 0;
    if (!grid) {
        int dev = 0, sms = 0, per = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, k_hash<4, false>, 256, 0);
        grid = sms * (per > 0 ? per : 1);
    }
    return grid;
}

template <bool kP2>
static cudaError_t launch_hash_t(const DevState &d, const dm_batch &b, int grid, cudaStream_t st) {
    switch (d.B) {
        case 4: DM_TRY(launch_pdl(k_hash<1, kP2>, grid, 256, 0, st, d, b.tokens)); break;
        case 8: DM_TRY(launch_pdl(k_hash<2, kP2>, grid, 256, 0, st, d, b.tokens)); break;
        case 16: DM_TRY(launch_pdl(k_hash<4, kP2>, grid, 256, 0, st, d, b.tokens)); break;
        case 32: DM_TRY(launch_pdl(k_hash<8, kP2>, grid, 256, 0, st, d, b.tokens)); break;
        case 64: DM_TRY(launch_pdl(k_hash<16, kP2>, grid, 256, 0, st, d, b.tokens)); break;
        default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

cudaError_t launch_hash(const DevState &d, const dm_batch &b, int grid, cudaStream_t st) {
    return d.ad_step ? launch_hash_t<true>(d, b, grid, st) : launch_hash_t<false>(d, b, grid, st);
}

// ---------------------------------------------------------------------------
// dm_hash_prompts: full cache keys of every block, plus the two positions.
__global__ void k_hash_keys(DevState d, uint32_t n, uint64_t *keys, uint64_t *key_off, uint64_t *pos) {
    if (has_err(d.err)) return;
    const int lane = threadIdx.x & 31;
    const uint32_t r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (r >= n) return;
    request_carries(d, r, lane);
    __syncwarp();
    const uint32_t nblk = d.r_nblk[r], s0 = d.r_segoff[r];
    const uint64_t bo = d.r_blkoff[r];
    for (uint32_t b = lane; b < nblk; b += 32)
        keys[bo + b] = cache_key(d.plocal[bo + b] + d.seg_carry[s0 + b / kSegBlocks], d.Sc);
    uint64_t p1, p2;
    route_positions(d, r, lane, p1, p2);
    if (lane == 0) {
        key_off[r] = bo;
        pos[2 * r] = p1;
        pos[2 * r + 1] = p2;
        if (r == n - 1) key_off[n] = bo + nblk;
    }
}

cudaError_t launch_hash_keys(const DevState &d, uint32_t n, uint64_t *keys, uint64_t *key_off,
                             uint64_t *pos, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    const uint32_t warps = 8;
    k_hash_keys<<<(n + warps - 1) / warps, warps * 32, 0, st>>>(d, n, keys, key_off, pos);
    return cudaGetLastError();
}

}  // namespace dm
